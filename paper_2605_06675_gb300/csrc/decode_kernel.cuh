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
//   scores^T[32 tok x 8 heads] = K_hat[32 x 128] . q^T      (mma m16n8k16)
//   online softmax in fp32 (log2 domain), P^T via movmatrix.trans
//   o^T[128 x 8 heads]       += V_hat^T[128 x 32] . P^T    (mma m16n8k16)
// The GQA group (g <= 8 query heads) is the MMA n dimension, so it is never
// padded to 16. Each warp streams its K and V block images through its own
// ring of shared-memory slots with cp.async, several entries ahead of use.
// Codes are stored in the MMA-fragment order of format.cuh: one AND of a
// word yields a register's two codes as exact fp16 subnormals c * 2^(E - 24)
// that enter the tensor cores undequantized. For the KIVI layouts
// (per-channel keys, per-token values) the group scales and 2^-E are folded
// into the small operand (q or P) or the output rows, and the zero-points are
// added by extra MMAs whose A operand is the meta image as read; the other
// layouts dequantize in registers (fp16 1024 exponent, one fp16x2 FMA).
// Split records are merged by decode_merge_kernel, a programmatic dependent
// launch of the split kernel.
#pragma once

#include <algorithm>
#include <atomic>

#include "format.cuh"
#include "rq_internal.cuh"

namespace rq {
namespace dk {

constexpr int kWarps = 4;                 // warps per split (a group; the merge kernel's CTA)
constexpr int kThreads = 32 * kWarps;
constexpr int kGroups = 4;                // split groups per decode CTA
constexpr int kPart = kD + 4;        // partial record: o[128], m (log2 domain), l, 2 pad (16-byte rows)
constexpr int kMaxHeads = 8;         // MMA n
constexpr int kRingBytes = 11264;    // per-warp ring of shared-memory slots
constexpr int kMaxSlots = 8;
constexpr int kQBytes = kMaxHeads * kD * 4;
constexpr int kSmemBytes = kQBytes + kWarps * kRingBytes;   // 49152: q table and rings of a split group
// a split group's shared memory: q table, rings, the warps' (m, l), two
// Lloyd-Max codebooks and two code-pair tables (52480 bytes, a multiple of 128)
constexpr int kGroupBytes = kSmemBytes + 2 * kWarps * kMaxHeads * 4 + 2 * 256 * 2 + 2 * 256 * 4;
constexpr int kSplitSmem = kGroups * kGroupBytes;            // per four-group CTA
static_assert(kGroupBytes % 128 == 0, "group areas start on 128-byte boundaries");
static_assert(kWarps * kMaxHeads * kD * 4 <= kWarps * kRingBytes, "merge buffer aliases rings");

struct DecodeArgs {
  const void* q;
  const uint8_t* packed;
  const uint8_t* bits;
  const uint64_t* offsets;
  const int8_t* signs;
  float* partial;            // [B][H_q][splits][132]
  const int32_t* n_rows;     // tokens attended per batch row (rq_decode_attention_rows) or null
  uint32_t* status;
  // split plan: (batch, kv head) units [0, u_lo) take s_lo splits of bps_lo
  // blocks, the others `splits` splits of bps blocks (splits = s_lo or
  // s_lo + 1; it is also the record stride per query row); splits are
  // numbered unit by unit, the s_lo-split units' (larger) ones first
  int layer, B, H, Hq, g, nblk, splits, bps, s_lo, bps_lo, u_lo, kg, vg, hadamard;
  int kq, vq;                // rq_quantizer of keys / values
  int early;                 // let the merge grid launch before the blocks (else after)
  int mix;                   // deal each CTA one split per quarter of the plan (else consecutive)
  LMBook lm;                 // RQ_LLOYDMAX codebooks
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

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(src));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N)); }
__device__ __forceinline__ void cp_async_wait_dyn(int n) {
  switch (n) {
    case 0: cp_async_wait<0>(); break;
    case 1: cp_async_wait<1>(); break;
    case 2: cp_async_wait<2>(); break;
    case 3: cp_async_wait<3>(); break;
    case 4: cp_async_wait<4>(); break;
    case 5: cp_async_wait<5>(); break;
    case 6: cp_async_wait<6>(); break;
    default: cp_async_wait<7>(); break;
  }
}

// 2^x with the MUFU approximation (x <= 0 or small; -inf gives 0)
__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint4 lds128(const uint8_t* p) {
  return *reinterpret_cast<const uint4*>(p);
}

// ------------------------------------------------------- code extraction ----
// The lane's 4*BW code words of one block image (16-byte piece i of lane L at
// byte 16*(32 i + L)); unit u's words are w[BW u .. BW u + BW - 1].
template <int BW>
__device__ __forceinline__ void lane_words(const uint8_t* img, int lane, uint32_t (&w)[4 * BW]) {
#pragma unroll
  for (int i = 0; i < BW; ++i) {
    const uint4 u = lds128(img + 16 * (32 * i + lane));
    w[4 * i + 0] = u.x;
    w[4 * i + 1] = u.y;
    w[4 * i + 2] = u.z;
    w[4 * i + 3] = u.w;
  }
}

constexpr uint32_t kMagic = 0x64006400u;      // fp16 1024.0 in both halves
constexpr float kTwo24 = 16777216.0f;         // codes enter the MMA as c * 2^(E - 24)

__device__ __forceinline__ uint32_t hfma2u(uint32_t x, uint32_t m, uint32_t a) {
  return h2u(__hfma2(u2h(x), u2h(m), u2h(a)));
}
__device__ __forceinline__ uint32_t hsub2u(uint32_t x, uint32_t y) {
  return h2u(__hsub2(u2h(x), u2h(y)));
}
__device__ __forceinline__ uint32_t hmul2u(uint32_t x, uint32_t y) {
  return h2u(__hmul2(u2h(x), u2h(y)));
}

// 2^-E in both fp16 halves (E <= 14)
__host__ __device__ constexpr uint32_t pow2_neg_h2(int E) {
  return (static_cast<uint32_t>(15 - E) << 10) * 0x00010001u;
}

// register (x, y) of unit u of the lane's words: c * 2^(E - 24) per half
template <int BW>
__device__ __forceinline__ uint32_t reg(const uint32_t (&w)[4 * BW], int u, int x, int y) {
  return fmt::extract<BW>(w + BW * u, x, y);
}

// dequantized pair s * c + z from an extracted register (layouts whose scale
// cannot be folded): the subnormal c * 2^E under the 1024 exponent, minus
// 1024 (exact), times m = s * 2^-E plus z (one rounding)
__device__ __forceinline__ uint32_t dequant(uint32_t sub, uint32_t m, uint32_t z2) {
  return hfma2u(hsub2u(sub | kMagic, kMagic), m, z2);
}

// Lloyd-Max pair: the two codes of an extracted register (at bit E of each
// half) looked up in the width's fp16 codebook (shared memory), scaled by m
// and shifted by z2 (one fp16x2 FMA)
// Widths up to 4 read both levels of a register at once from a table of
// code pairs (entry c0 + 2^BW c1 = the fp16x2 pair (L_c0, L_c1)): one
// shared-memory read per register instead of two; `tab` then points to it.
template <int BW>
__device__ __forceinline__ uint32_t lm_pair(uint32_t sub, int E, const uint16_t* tab) {
  const uint32_t c0 = (sub >> E) & ((1u << BW) - 1u), c1 = (sub >> (16 + E)) & ((1u << BW) - 1u);
  if constexpr (BW <= 4) return reinterpret_cast<const uint32_t*>(tab)[c0 | (c1 << BW)];
  else return static_cast<uint32_t>(tab[c0]) | (static_cast<uint32_t>(tab[c1]) << 16);
}

// ------------------------------------------------------------ block math ----
// Lane (gid, tig) reads units u = 0..3 of its K words: unit u holds channels
// 32 u + 8 tig + (0..7) of tokens gid + 8 (0..3); the k-steps 2u and 2u + 1
// of the scores MMA are its channel pairs x = 0, 1 and 2, 3 (format.cuh).
//
// scores^T[mt] (tokens 16 mt + gid (+8), heads 2 tig (+1)) of one K block image.
// Per-channel keys: k_hat[t][c] = code s_c + z_c, so
//   scores[t][j] = sum_c code[t][c] (q_jc s_c) + sum_c z_c q_jc:
// the scale (and the code's 2^-E) is folded into q, one fp16x2 multiply per
// q pair; the zero-point term, the same for every token, comes from MMAs
// whose A operand carries z in rows gid. Codes enter the tensor cores as
// exact fp16 subnormals c 2^(E - 24); the accumulator is scaled by 2^24.
// q operands of lane L for unit u: qtab + 16 (32 u + L) holds q pairs x = 0..3
// (channels 32u + 8tig + 2x), qtab + 2048 + the same with 2^-E(x) folded in.
// s is returned in log2 units (q . k times qsc = log2(e) / sqrt(128), applied
// here in fp32 so q enters the MMAs unscaled) relative to the running max
// (ms0, ms1: the max of heads 2tig, 2tig + 1, 0 while unset).
// q s 2^-E enters as an fp16 sum hi + lo (lo = the exact remainder, one fp16
// FMA), so the products keep ~22 bits. With g <= 4 query heads (MERGED)
// the MMA's 8 columns hold hi for heads 0..3 and lo for the same heads in
// columns 4..7 (lanes gid >= 4 carry q of head gid - 4 and mneg = -1 there,
// -0 elsewhere), and one shuffle adds the halves; otherwise hi and lo take
// one MMA each.
template <int BW, int KG, bool MERGED, bool LM = false>
__device__ __forceinline__ void qk_block(const uint8_t* img, int lane, const uint8_t* qtab,
                                         float qsc, float ms0, float ms1, uint32_t mneg,
                                         float (&s)[2][4], const uint16_t* lmtab = nullptr) {
  const int gid = lane >> 2, tig = lane & 3;
  uint32_t w[4 * BW];
  lane_words<BW>(img, lane, w);
  const uint8_t* meta = img + 512 * BW;
#pragma unroll
  for (int mt = 0; mt < 2; ++mt)
#pragma unroll
    for (int r = 0; r < 4; ++r) s[mt][r] = 0.0f;
  if constexpr (KG == RQ_PER_CHANNEL) {
    float zb[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      // channel pairs P = 16u + 4tig + x: zeros at word 2P, scales at 2P + 1,
      // so each 16-byte read {z(x), s(x), z(x+1), s(x+1)} is the A operand of
      // a zero-point MMA (rows gid take z; rows gid + 8 take s and are unused)
      const uint4 MZ0 = lds128(meta + 4 * (32 * u + 8 * tig));
      const uint4 MZ1 = lds128(meta + 4 * (32 * u + 8 * tig + 4));
      const uint4 QB = lds128(qtab + 16 * (32 * u + lane));
      const uint4 QF = lds128(qtab + 2048 + 16 * (32 * u + lane));
      const uint32_t qb[4] = {QB.x, QB.y, QB.z, QB.w}, qf[4] = {QF.x, QF.y, QF.z, QF.w};
#pragma unroll
      for (int xs = 0; xs < 2; ++xs) {
        const uint4 MZ = xs ? MZ1 : MZ0;
        const uint32_t h0 = hmul2u(qf[2 * xs], MZ.y);
        const uint32_t h1 = hmul2u(qf[2 * xs + 1], MZ.w);
        const uint32_t az[4] = {MZ.x, MZ.y, MZ.z, MZ.w};
        mma16816(zb, az, qb[2 * xs], qb[2 * xs + 1]);
        if constexpr (MERGED) {
          // hi lanes: fma(q, s, hi * -0) = hi; lo lanes: fma(q, s, -hi) = lo
          // (fp16 multiplies, not bitwise ops: they run on the FMA pipe,
          // which the code extraction leaves idle)
          const uint32_t b0 = hfma2u(qf[2 * xs], MZ.y, hmul2u(h0, mneg));
          const uint32_t b1 = hfma2u(qf[2 * xs + 1], MZ.w, hmul2u(h1, mneg));
#pragma unroll
          for (int mt = 0; mt < 2; ++mt) {
            const uint32_t a[4] = {reg<BW>(w, u, 2 * xs, 2 * mt), reg<BW>(w, u, 2 * xs, 2 * mt + 1),
                                   reg<BW>(w, u, 2 * xs + 1, 2 * mt), reg<BW>(w, u, 2 * xs + 1, 2 * mt + 1)};
            mma16816(s[mt], a, b0, b1);
          }
        } else {
          const uint32_t l0 = hfma2u(qf[2 * xs], MZ.y, h0 ^ 0x80008000u);
          const uint32_t l1 = hfma2u(qf[2 * xs + 1], MZ.w, h1 ^ 0x80008000u);
#pragma unroll
          for (int mt = 0; mt < 2; ++mt) {
            const uint32_t a[4] = {reg<BW>(w, u, 2 * xs, 2 * mt), reg<BW>(w, u, 2 * xs, 2 * mt + 1),
                                   reg<BW>(w, u, 2 * xs + 1, 2 * mt), reg<BW>(w, u, 2 * xs + 1, 2 * mt + 1)};
            mma16816(s[mt], a, h0, h1);
            mma16816(s[mt], a, l0, l1);
          }
        }
      }
    }
    if constexpr (MERGED) {   // columns j and j + 4 of the accumulator: hi + lo
#pragma unroll
      for (int mt = 0; mt < 2; ++mt)
#pragma unroll
        for (int r = 0; r < 4; ++r) s[mt][r] += __shfl_xor_sync(0xffffffffu, s[mt][r], 2);
    }
    const float c0 = __fmaf_rn(zb[0], qsc, -ms0), c1 = __fmaf_rn(zb[1], qsc, -ms1);
    const float f = kTwo24 * qsc;
#pragma unroll
    for (int mt = 0; mt < 2; ++mt) {
      s[mt][0] = __fmaf_rn(s[mt][0], f, c0);
      s[mt][1] = __fmaf_rn(s[mt][1], f, c1);
      s[mt][2] = __fmaf_rn(s[mt][2], f, c0);
      s[mt][3] = __fmaf_rn(s[mt][3], f, c1);
    }
  } else if constexpr (!LM) {
    // Per-token keys: k_hat[t][c] = code s_tG + z_tG, so for group G = unit u
    //   scores[t][j] += s_tG sum_{c in G} code[t][c] q_jc + z_tG sum_{c in G} q_jc:
    // the codes enter the MMA undequantized (two k-steps per group into a
    // group accumulator), and the group's scale (with the codes' 2^(24 - E)
    // of the token row) and zero term are applied to that accumulator in fp32.
    // qsum (the QF area of the table) holds sum_{c in G} q_jc for [G][head].
    const float* qsum = reinterpret_cast<const float*>(qtab + 2048);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      // (scale, zero) of tokens 8x + gid, group u: words 16 gid + 4u + x
      const uint4 SZ = lds128(meta + 4 * (16 * gid + 4 * u));
      const uint4 QB = lds128(qtab + 16 * (32 * u + lane));
      const float2 qs = *reinterpret_cast<const float2*>(qsum + 8 * u + 2 * tig);
      const uint32_t qb[4] = {QB.x, QB.y, QB.z, QB.w};
      const uint32_t sz[4] = {SZ.x, SZ.y, SZ.z, SZ.w};
      float acc[2][4];
#pragma unroll
      for (int mt = 0; mt < 2; ++mt)
#pragma unroll
        for (int r = 0; r < 4; ++r) acc[mt][r] = 0.0f;
#pragma unroll
      for (int xs = 0; xs < 2; ++xs)
#pragma unroll
        for (int mt = 0; mt < 2; ++mt) {
          // register (x = token 2mt + r, y = pair 2xs + h)
          const uint32_t a[4] = {reg<BW>(w, u, 2 * mt, 2 * xs), reg<BW>(w, u, 2 * mt + 1, 2 * xs),
                                 reg<BW>(w, u, 2 * mt, 2 * xs + 1), reg<BW>(w, u, 2 * mt + 1, 2 * xs + 1)};
          mma16816(acc[mt], a, qb[2 * xs], qb[2 * xs + 1]);
        }
#pragma unroll
      for (int mt = 0; mt < 2; ++mt) {
        // rows gid / gid + 8: tokens of class x = 2mt / 2mt + 1
        const __half2 h0 = u2h(sz[2 * mt]), h1 = u2h(sz[2 * mt + 1]);
        const float s0 = __fmul_rn(__low2float(h0), __int_as_float((127 + 24 - fmt::exponent(BW, 2 * mt)) << 23));
        const float s1 = __fmul_rn(__low2float(h1), __int_as_float((127 + 24 - fmt::exponent(BW, 2 * mt + 1)) << 23));
        const float z0 = __high2float(h0), z1 = __high2float(h1);
        s[mt][0] = __fmaf_rn(acc[mt][0], s0, __fmaf_rn(z0, qs.x, s[mt][0]));
        s[mt][1] = __fmaf_rn(acc[mt][1], s0, __fmaf_rn(z0, qs.y, s[mt][1]));
        s[mt][2] = __fmaf_rn(acc[mt][2], s1, __fmaf_rn(z1, qs.x, s[mt][2]));
        s[mt][3] = __fmaf_rn(acc[mt][3], s1, __fmaf_rn(z1, qs.y, s[mt][3]));
      }
    }
#pragma unroll
    for (int mt = 0; mt < 2; ++mt) {
      s[mt][0] = __fmaf_rn(s[mt][0], qsc, -ms0);
      s[mt][1] = __fmaf_rn(s[mt][1], qsc, -ms1);
      s[mt][2] = __fmaf_rn(s[mt][2], qsc, -ms0);
      s[mt][3] = __fmaf_rn(s[mt][3], qsc, -ms1);
    }
  } else {                    // Lloyd-Max per-token keys: codebook levels in registers
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      // (scale, zero) of tokens 8x + gid, group u: words 16 gid + 4u + x
      const uint4 SZ = lds128(meta + 4 * (16 * gid + 4 * u));
      const uint4 QB = lds128(qtab + 16 * (32 * u + lane));
      const uint32_t qb[4] = {QB.x, QB.y, QB.z, QB.w};
      const uint32_t sz[4] = {SZ.x, SZ.y, SZ.z, SZ.w};
      uint32_t m[4], z2[4];
#pragma unroll
      for (int x = 0; x < 4; ++x) {
        const __half2 h = u2h(sz[x]);
        m[x] = LM ? h2u(__low2half2(h))          // codebook levels are real values
                  : hmul2u(h2u(__low2half2(h)), pow2_neg_h2(fmt::exponent(BW, x)));
        z2[x] = h2u(__high2half2(h));
      }
      auto deq = [&](int x, int y) -> uint32_t {
        if constexpr (LM) return hfma2u(lm_pair<BW>(reg<BW>(w, u, x, y), fmt::exponent(BW, x), lmtab),
                                        m[x], z2[x]);
        else return dequant(reg<BW>(w, u, x, y), m[x], z2[x]);
      };
#pragma unroll
      for (int xs = 0; xs < 2; ++xs)
#pragma unroll
        for (int mt = 0; mt < 2; ++mt) {
          // register (x = token 2mt + r, y = pair 2xs + h)
          const uint32_t a[4] = {deq(2 * mt, 2 * xs), deq(2 * mt + 1, 2 * xs),
                                 deq(2 * mt, 2 * xs + 1), deq(2 * mt + 1, 2 * xs + 1)};
          mma16816(s[mt], a, qb[2 * xs], qb[2 * xs + 1]);
        }
    }
#pragma unroll
    for (int mt = 0; mt < 2; ++mt) {
      s[mt][0] = __fmaf_rn(s[mt][0], qsc, -ms0);
      s[mt][1] = __fmaf_rn(s[mt][1], qsc, -ms1);
      s[mt][2] = __fmaf_rn(s[mt][2], qsc, -ms0);
      s[mt][3] = __fmaf_rn(s[mt][3], qsc, -ms1);
    }
  }
}

// o^T[mt] (channel rows 16 mt + gid (+8), heads 2 tig (+1)) += V_hat^T . P^T of
// one V block image. Unit u = channel group G holds channels 32u + 4gid + x
// (rows of m-tiles 2u, 2u + 1) of tokens 8y + 2tig + (0, 1).
// Per-token values: v_hat[t][c] = code s_tG + z_tG, so
//   o[c][j] += sum_t code[t][c] (p_tj s_tG) + sum_t z_tG p_tj:
// the scale is folded into P^T per group (one fp16x2 multiply per pair), the
// zero-point term comes from MMAs whose A operand repeats z_tG in every row
// of the group, and the codes' 2^(E - 24) is undone on the output rows.
template <int BW, int VG, bool LM = false>
__device__ __forceinline__ void pv_block(const uint8_t* img, int lane, const uint32_t (&pb)[2][2],
                                         float (&o)[8][4], float (&bz)[2][4],
                                         const uint16_t* lmtab = nullptr) {
  const int gid = lane >> 2, tig = lane & 3;
  uint32_t w[4 * BW];
  lane_words<BW>(img, lane, w);
  const uint8_t* meta = img + 512 * BW;
  if constexpr (VG == RQ_PER_TOKEN) {
    // zero-points: rows gid of the A operand carry group 2gp, rows gid + 8
    // group 2gp + 1; columns are token pairs 2ks (k 2tig..) and 2ks + 1.
    // Zero pairs are stored so that each 16-byte read is an A operand:
    // words 64 + 32ks + 8tig + 4gp + {0..3} = z of (token pair 2ks, group
    // 2gp), (2ks, 2gp+1), (2ks+1, 2gp), (2ks+1, 2gp+1).
#pragma unroll
    for (int ks = 0; ks < 2; ++ks)
#pragma unroll
      for (int gp = 0; gp < 2; ++gp) {
        const uint4 Z = lds128(meta + 4 * (64 + 32 * ks + 8 * tig + 4 * gp));
        const uint32_t az[4] = {Z.x, Z.y, Z.z, Z.w};
        mma16816(bz[gp], az, pb[ks][0], pb[ks][1]);
      }
    uint32_t ms[4][4];        // scale pairs [token pair y][group G]: words 16y + 4tig + G
#pragma unroll
    for (int y = 0; y < 4; ++y) {
      const uint4 S = lds128(meta + 4 * (16 * y + 4 * tig));
      ms[y][0] = S.x;
      ms[y][1] = S.y;
      ms[y][2] = S.z;
      ms[y][3] = S.w;
    }
#pragma unroll
    for (int ks = 0; ks < 2; ++ks)
#pragma unroll
      for (int G = 0; G < 4; ++G) {
        const uint32_t b0 = hmul2u(pb[ks][0], ms[2 * ks][G]);
        const uint32_t b1 = hmul2u(pb[ks][1], ms[2 * ks + 1][G]);
#pragma unroll
        for (int mh = 0; mh < 2; ++mh) {
          // register (x = row 2mh + r, y = token pair 2ks + h); Lloyd-Max: the
          // codebook levels (real values) instead of the subnormal codes
          auto A = [&](int x, int y) -> uint32_t {
            if constexpr (LM) return lm_pair<BW>(reg<BW>(w, G, x, y), fmt::exponent(BW, x), lmtab);
            else return reg<BW>(w, G, x, y);
          };
          const uint32_t a[4] = {A(2 * mh, 2 * ks), A(2 * mh + 1, 2 * ks), A(2 * mh, 2 * ks + 1),
                                 A(2 * mh + 1, 2 * ks + 1)};
          mma16816(o[2 * G + mh], a, b0, b1);
        }
      }
  } else {                    // per-channel values: dequantize in registers
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      // (scale, zero) of channels 32u + 4gid + x: words 32u + 4gid + x
      const uint4 SZ = lds128(meta + 4 * (32 * u + 4 * gid));
      const uint32_t sz[4] = {SZ.x, SZ.y, SZ.z, SZ.w};
      uint32_t m[4], z2[4];
#pragma unroll
      for (int x = 0; x < 4; ++x) {
        const __half2 h = u2h(sz[x]);
        m[x] = hmul2u(h2u(__low2half2(h)), pow2_neg_h2(fmt::exponent(BW, x)));
        z2[x] = h2u(__high2half2(h));
      }
#pragma unroll
      for (int ks = 0; ks < 2; ++ks)
#pragma unroll
        for (int mh = 0; mh < 2; ++mh) {
          const uint32_t a[4] = {
              dequant(reg<BW>(w, u, 2 * mh, 2 * ks), m[2 * mh], z2[2 * mh]),
              dequant(reg<BW>(w, u, 2 * mh + 1, 2 * ks), m[2 * mh + 1], z2[2 * mh + 1]),
              dequant(reg<BW>(w, u, 2 * mh, 2 * ks + 1), m[2 * mh], z2[2 * mh]),
              dequant(reg<BW>(w, u, 2 * mh + 1, 2 * ks + 1), m[2 * mh + 1], z2[2 * mh + 1])};
          mma16816(o[2 * u + mh], a, pb[ks][0], pb[ks][1]);
        }
    }
  }
}

template <int BW>
__device__ __forceinline__ void qk_dispatch_g(int kg, const uint8_t* img, int lane,
                                              const uint8_t* qtab, float qsc, float ms0, float ms1,
                                              float (&s)[2][4], const uint16_t* lmtab) {
  // mneg is unused off the merged path; lmtab is non-null for Lloyd-Max keys
  if (kg == RQ_PER_CHANNEL) qk_block<BW, RQ_PER_CHANNEL, false>(img, lane, qtab, qsc, ms0, ms1, 0u, s);
  else if (lmtab) qk_block<BW, RQ_PER_TOKEN, false, true>(img, lane, qtab, qsc, ms0, ms1, 0u, s, lmtab);
  else qk_block<BW, RQ_PER_TOKEN, false>(img, lane, qtab, qsc, ms0, ms1, 0u, s);
}

template <int BW>
__device__ __forceinline__ void pv_dispatch_g(int vg, const uint8_t* img, int lane,
                                              const uint32_t (&pb)[2][2], float (&o)[8][4],
                                              float (&bz)[2][4], const uint16_t* lmtab) {
  if (vg == RQ_PER_TOKEN && lmtab) pv_block<BW, RQ_PER_TOKEN, true>(img, lane, pb, o, bz, lmtab);
  else if (vg == RQ_PER_TOKEN) pv_block<BW, RQ_PER_TOKEN>(img, lane, pb, o, bz);
  else pv_block<BW, RQ_PER_CHANNEL>(img, lane, pb, o, bz);
}

__device__ __forceinline__ void qk_dispatch(int bw, int kg, const uint8_t* img, int lane,
                                            const uint8_t* qtab, float qsc, float ms0, float ms1,
                                            float (&s)[2][4], const uint16_t* lmtab) {
  switch (bw) {
    case 1: qk_dispatch_g<1>(kg, img, lane, qtab, qsc, ms0, ms1, s, lmtab); break;
    case 2: qk_dispatch_g<2>(kg, img, lane, qtab, qsc, ms0, ms1, s, lmtab); break;
    case 3: qk_dispatch_g<3>(kg, img, lane, qtab, qsc, ms0, ms1, s, lmtab); break;
    case 4: qk_dispatch_g<4>(kg, img, lane, qtab, qsc, ms0, ms1, s, lmtab); break;
    case 5: qk_dispatch_g<5>(kg, img, lane, qtab, qsc, ms0, ms1, s, lmtab); break;
    case 6: qk_dispatch_g<6>(kg, img, lane, qtab, qsc, ms0, ms1, s, lmtab); break;
    case 7: qk_dispatch_g<7>(kg, img, lane, qtab, qsc, ms0, ms1, s, lmtab); break;
    default: qk_dispatch_g<8>(kg, img, lane, qtab, qsc, ms0, ms1, s, lmtab); break;
  }
}

__device__ __forceinline__ void pv_dispatch(int bw, int vg, const uint8_t* img, int lane,
                                            const uint32_t (&pb)[2][2], float (&o)[8][4],
                                            float (&bz)[2][4], const uint16_t* lmtab) {
  switch (bw) {
    case 1: pv_dispatch_g<1>(vg, img, lane, pb, o, bz, lmtab); break;
    case 2: pv_dispatch_g<2>(vg, img, lane, pb, o, bz, lmtab); break;
    case 3: pv_dispatch_g<3>(vg, img, lane, pb, o, bz, lmtab); break;
    case 4: pv_dispatch_g<4>(vg, img, lane, pb, o, bz, lmtab); break;
    case 5: pv_dispatch_g<5>(vg, img, lane, pb, o, bz, lmtab); break;
    case 6: pv_dispatch_g<6>(vg, img, lane, pb, o, bz, lmtab); break;
    case 7: pv_dispatch_g<7>(vg, img, lane, pb, o, bz, lmtab); break;
    default: pv_dispatch_g<8>(vg, img, lane, pb, o, bz, lmtab); break;
  }
}

// 128-point FWHT of each of `rows` rows of x (row stride 128), strides 1..64
// named barrier of split group grp (kThreads threads; barrier 0 is the
// CTA's). Immediate barrier ids: a register id would reserve all 16 of the
// CTA's barriers.
__device__ __forceinline__ void group_sync(int grp) {
  switch (grp) {
    case 0: asm volatile("bar.sync 1, %0;\n" ::"n"(kThreads) : "memory"); break;
    case 1: asm volatile("bar.sync 2, %0;\n" ::"n"(kThreads) : "memory"); break;
    case 2: asm volatile("bar.sync 3, %0;\n" ::"n"(kThreads) : "memory"); break;
    default: asm volatile("bar.sync 4, %0;\n" ::"n"(kThreads) : "memory"); break;
  }
}
static_assert(kGroups == 4, "group_sync names four barriers");

// fwht_smem for one split group: thread tl of group grp
__device__ inline void fwht_smem_group(float* x, int rows, int tl, int grp) {
  for (int lh = 0; lh < 7; ++lh) {
    const int h = 1 << lh;
    for (int p = tl; p < rows * 64; p += kThreads) {
      const int row = p >> 6, pi = p & 63;
      const int i = ((pi >> lh) << (lh + 1)) | (pi & (h - 1));
      float* r = x + row * kD;
      const float a = r[i], b = r[i + h];
      r[i] = a + b;
      r[i + h] = a - b;
    }
    group_sync(grp);
  }
}

__device__ inline void fwht_smem(float* x, int rows) {
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

// Issue the cp.async copies of one ring entry (the K or V image of one
// block, `bytes` long, at `src`) into the slot at shared address `dst`; one
// commit group per entry (empty when there is nothing left, so the group
// count stays uniform).
__device__ __forceinline__ void issue_entry(bool live, int lane, uint32_t dst, const uint8_t* src,
                                            int bytes) {
  if (live) {
    const int chunks = bytes >> 4;
    for (int ch = lane; ch < chunks; ch += 32) cp_async16(dst + 16 * ch, src + 16 * ch);
  }
  cp_async_commit();
}

// Per-warp streaming state: the warp's blocks are blk_first, blk_first + 4,
// ... of one (batch, kv head) K and V stream; ring entry e is the K image
// (e even) or V image (e odd) of the warp's block e / 2.
struct WarpStream {
  const uint8_t* kwarp;   // K image of the warp's first block
  const uint8_t* vwarp;
  uint8_t* ring_ptr;      // this warp's ring of slots
  uint32_t ring;          // its shared-memory address
  int lane, nb;
  bool merged;            // g <= 4: hi and lo q operands share one MMA
  uint32_t mneg;          // merged: fp16x2 -1 on the lanes that carry lo (gid >= 4), else -0
};

// online-softmax state of one warp: o^T accumulators and per-column max/sum
struct SoftmaxAcc {
  float o[8][4];
  float bz[2][4];   // per-token V zero-point sums: rows gid -> groups 0/2, rows gid+8 -> 1/3
  float m0, m1, l0, l1;
};

// softmax of one block's scores (log2 units) into the accumulator; returns
// the B fragments of P^T. The running max only moves when a block max
// exceeds it by more than 8, so p <= 2^8 and rescaling is rare.
__device__ __forceinline__ void softmax_block(float (&s)[2][4], SoftmaxAcc& acc,
                                              uint32_t (&pb)[2][2]) {
  // s holds score - running max (log2 units). Each lane checks its own
  // values; only when one exceeds the bound is the column max reduced across
  // the lanes and the running max moved (rare), so p <= 2^8 always.
  float bm0 = fmaxf(fmaxf(s[0][0], s[0][2]), fmaxf(s[1][0], s[1][2]));
  float bm1 = fmaxf(fmaxf(s[0][1], s[0][3]), fmaxf(s[1][1], s[1][3]));
  const bool first = acc.m0 == -INFINITY;      // the warp's first block: set the max
  if (__any_sync(0xffffffffu, first || bm0 > 8.0f || bm1 > 8.0f)) {
#pragma unroll
    for (int off = 4; off <= 16; off <<= 1) {
      bm0 = fmaxf(bm0, __shfl_xor_sync(0xffffffffu, bm0, off));
      bm1 = fmaxf(bm1, __shfl_xor_sync(0xffffffffu, bm1, off));
    }
    // first block: max = block max (s holds raw scores); later: the max moves
    // up by d = max(block max - m, 0) and the state is scaled by 2^-d
    float d0, d1, al0, al1;
    if (first) {
      d0 = bm0;
      d1 = bm1;
      al0 = al1 = 0.0f;
      acc.m0 = bm0;
      acc.m1 = bm1;
    } else {
      d0 = fmaxf(bm0, 0.0f);
      d1 = fmaxf(bm1, 0.0f);
      al0 = fast_exp2(-d0);
      al1 = fast_exp2(-d1);
      acc.m0 += d0;
      acc.m1 += d1;
    }
#pragma unroll
    for (int mt = 0; mt < 2; ++mt) {
      s[mt][0] -= d0;
      s[mt][1] -= d1;
      s[mt][2] -= d0;
      s[mt][3] -= d1;
    }
    acc.l0 *= al0;
    acc.l1 *= al1;
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) {
      acc.o[mt][0] *= al0;
      acc.o[mt][1] *= al1;
      acc.o[mt][2] *= al0;
      acc.o[mt][3] *= al1;
    }
#pragma unroll
    for (int gp = 0; gp < 2; ++gp) {
      acc.bz[gp][0] *= al0;
      acc.bz[gp][1] *= al1;
      acc.bz[gp][2] *= al0;
      acc.bz[gp][3] *= al1;
    }
  }
  float p[2][4];
#pragma unroll
  for (int mt = 0; mt < 2; ++mt)
#pragma unroll
    for (int r = 0; r < 4; ++r) p[mt][r] = fast_exp2(s[mt][r]);
  acc.l0 += (p[0][0] + p[0][2]) + (p[1][0] + p[1][2]);
  acc.l1 += (p[0][1] + p[0][3]) + (p[1][1] + p[1][3]);
#pragma unroll
  for (int ks = 0; ks < 2; ++ks) {
    pb[ks][0] = movmatrix_trans(pack_f16x2(p[ks][0], p[ks][1]));
    pb[ks][1] = movmatrix_trans(pack_f16x2(p[ks][2], p[ks][3]));
  }
}

// ---- streaming with widths and groupings fixed at compile time: slot sizes,
// slot counts, copy counts and the wait depth are constants, and the fp16
// constants of the code extraction stay in registers across the loop.
template <int BK, int BV>
struct Ring {
  static constexpr int kSK = 512 * (BK + 1), kSV = 512 * (BV + 1);
  static constexpr int kSlot = kSK > kSV ? kSK : kSV;
  static constexpr int kRaw = kRingBytes / kSlot;
  static constexpr int kSlots = kRaw > kMaxSlots ? kMaxSlots : kRaw;
};

template <int BK, int BV>
__device__ __forceinline__ void issue_static(const WarpStream& ws, int e, int slot) {
  using R = Ring<BK, BV>;
  if (e < 2 * ws.nb) {
    const int i = e >> 1;
    const uint32_t dst = ws.ring + slot * R::kSlot;
    if ((e & 1) == 0) {
      const uint8_t* src = ws.kwarp + i * (kWarps * R::kSK);
#pragma unroll
      for (int c = 0; c < R::kSK / 512; ++c) cp_async16(dst + 16 * (ws.lane + 32 * c), src + 16 * (ws.lane + 32 * c));
    } else {
      const uint8_t* src = ws.vwarp + i * (kWarps * R::kSV);
#pragma unroll
      for (int c = 0; c < R::kSV / 512; ++c) cp_async16(dst + 16 * (ws.lane + 32 * c), src + 16 * (ws.lane + 32 * c));
    }
  }
  cp_async_commit();
}

template <int BK, int BV>
__device__ __forceinline__ void prologue_static(const WarpStream& ws) {
#pragma unroll
  for (int e = 0; e < Ring<BK, BV>::kSlots - 1; ++e) issue_static<BK, BV>(ws, e, e);
}

template <int BK, int KG, int BV, int VG, bool MERGED>
__device__ __forceinline__ void blocks_static(const WarpStream& ws, const uint8_t* qtab, float qsc,
                                              SoftmaxAcc& acc) {
  using R = Ring<BK, BV>;
  constexpr int NS = R::kSlots;
  int use = 0, iss = NS - 1;          // slot of the next entry to use / to issue
  for (int i = 0; i < ws.nb; ++i) {
    issue_static<BK, BV>(ws, 2 * i + NS - 1, iss);
    iss = iss + 1 == NS ? 0 : iss + 1;
    cp_async_wait<NS - 1>();
    __syncwarp();
    float s[2][4];
    qk_block<BK, KG, MERGED>(ws.ring_ptr + use * R::kSlot, ws.lane, qtab, qsc,
                     acc.m0 == -INFINITY ? 0.0f : acc.m0, acc.m1 == -INFINITY ? 0.0f : acc.m1,
                     ws.mneg, s);
    __syncwarp();
    use = use + 1 == NS ? 0 : use + 1;
    uint32_t pb[2][2];
    softmax_block(s, acc, pb);
    issue_static<BK, BV>(ws, 2 * i + NS, iss);
    iss = iss + 1 == NS ? 0 : iss + 1;
    cp_async_wait<NS - 1>();
    __syncwarp();
    pv_block<BV, VG>(ws.ring_ptr + use * R::kSlot, ws.lane, pb, acc.o, acc.bz);
    __syncwarp();
    use = use + 1 == NS ? 0 : use + 1;
  }
  cp_async_wait<0>();
}

// ---- streaming with runtime widths/groupings (every other combination)
struct DynRing {
  int bK, bV, kg, vg, sK, sV, slot, ns;
  const uint16_t* lmK;       // Lloyd-Max codebook of the key / value width (null: none)
  const uint16_t* lmV;
};

__device__ __forceinline__ void issue_dyn(const WarpStream& ws, const DynRing& r, int e, int slot) {
  const int i = e >> 1;
  const bool isK = (e & 1) == 0;
  issue_entry(e < 2 * ws.nb, ws.lane, ws.ring + slot * r.slot,
              isK ? ws.kwarp + i * (kWarps * r.sK) : ws.vwarp + i * (kWarps * r.sV), isK ? r.sK : r.sV);
}

__device__ __forceinline__ void prologue_dyn(const WarpStream& ws, const DynRing& r) {
  for (int e = 0; e < r.ns - 1; ++e) issue_dyn(ws, r, e, e);
}

__device__ __forceinline__ void blocks_dyn(const WarpStream& ws, const DynRing& r,
                                           const uint8_t* qtab, float qsc, SoftmaxAcc& acc) {
  int use = 0, iss = r.ns - 1;
  for (int i = 0; i < ws.nb; ++i) {
    issue_dyn(ws, r, 2 * i + r.ns - 1, iss);
    iss = iss + 1 == r.ns ? 0 : iss + 1;
    cp_async_wait_dyn(r.ns - 1);
    __syncwarp();
    float s[2][4];
    qk_dispatch(r.bK, r.kg, ws.ring_ptr + use * r.slot, ws.lane, qtab, qsc,
                acc.m0 == -INFINITY ? 0.0f : acc.m0, acc.m1 == -INFINITY ? 0.0f : acc.m1, s, r.lmK);
    __syncwarp();
    use = use + 1 == r.ns ? 0 : use + 1;
    uint32_t pb[2][2];
    softmax_block(s, acc, pb);
    issue_dyn(ws, r, 2 * i + r.ns, iss);
    iss = iss + 1 == r.ns ? 0 : iss + 1;
    cp_async_wait_dyn(r.ns - 1);
    __syncwarp();
    pv_dispatch(r.bV, r.vg, ws.ring_ptr + use * r.slot, ws.lane, pb, acc.o, acc.bz, r.lmV);
    __syncwarp();
    use = use + 1 == r.ns ? 0 : use + 1;
  }
  cp_async_wait<0>();
}

// Key of the compile-time path, or -1: keys 0..15 for the KIVI layout
// (per-channel K, per-token V) at widths {2, 3, 4, 8}; keys 16..31 for
// per-token K and V (the rotated caches) at key widths 3..6 and value widths
// 2..5, the widths an allocation at about 4 bits per code gives (keys take
// the wider ones).
__device__ __forceinline__ int fast_key(int bK, int bV, int kg, int vg) {
  if (kg == RQ_PER_CHANNEL && vg == RQ_PER_TOKEN) {
    auto idx = [](int b) { return b == 2 ? 0 : b == 3 ? 1 : b == 4 ? 2 : b == 8 ? 3 : -1; };
    const int ik = idx(bK), iv = idx(bV);
    return (ik < 0 || iv < 0) ? -1 : 4 * ik + iv;
  }
  if (kg == RQ_PER_TOKEN && vg == RQ_PER_TOKEN) {
    const int ik = bK >= 3 && bK <= 6 ? bK - 3 : -1, iv = bV >= 2 && bV <= 5 ? bV - 2 : -1;
    return (ik < 0 || iv < 0) ? -1 : 16 + 4 * ik + iv;
  }
  return -1;
}

#define RQ_FAST_CASES(X) \
  X(0, 2, 2) X(1, 2, 3) X(2, 2, 4) X(3, 2, 8) X(4, 3, 2) X(5, 3, 3) X(6, 3, 4) X(7, 3, 8) \
  X(8, 4, 2) X(9, 4, 3) X(10, 4, 4) X(11, 4, 8) X(12, 8, 2) X(13, 8, 3) X(14, 8, 4) X(15, 8, 8)
#define RQ_TOKEN_CASES(X) \
  X(16, 3, 2) X(17, 3, 3) X(18, 3, 4) X(19, 3, 5) X(20, 4, 2) X(21, 4, 3) X(22, 4, 4) X(23, 4, 5) \
  X(24, 5, 2) X(25, 5, 3) X(26, 5, 4) X(27, 5, 5) X(28, 6, 2) X(29, 6, 3) X(30, 6, 4) X(31, 6, 5)

// Two register budgets for the same code (the body below is included in
// both). At 128 registers a thread the split CTAs of an SM take all 65,536
// of its registers, so a merge CTA starts on an SM only where a split CTA has
// left. At 120 (28 bytes of spill stores), 4,096 stay free on every SM: one
// merge CTA of 128 threads at <= 32 registers fits beside the split CTAs
// when its shared memory does too, and waits there for the split grid to
// end. (A launch bound of 512 threads on the 120-register kernel, or the body
// as an inlined function, made the compiler spill several times more.)
template <typename T>
__global__ void __launch_bounds__(kThreads * kGroups, 1) decode_split_kernel(DecodeArgs a) {
#include "decode_split_body.inc"
}
template <typename T>
__global__ void __maxnreg__(120) decode_split_kernel_co(DecodeArgs a) {
#include "decode_split_body.inc"
}

// ------------------------------------------------------------ split merge ----
// out_n = sum_s 2^(m_ns - M_n) o_ns / sum_s 2^(m_ns - M_n) l_ns for the g
// query rows n of one (batch, kv head), rotated back (o R^T =
// FWHT(o) / sqrt(128) * signs) for a Hadamard cache. A CTA owns one (batch,
// kv head) and 128 / CQ channels of its rows (the whole row when CQ = 1, as
// the rotation needs). It is launched as a programmatic dependent of the
// split kernel and waits for it on entry. Records are pulled into shared
// memory with cp.async, a chunk of splits at a time (one round trip per
// chunk), and merged there with a running max per row.
constexpr int kMergeSmem = 64 * 1024;
constexpr int kMergeChunk = 128;     // split records merged per round trip, at most

// The unquantized residual tokens (decode-time append) of one (batch, kv
// head): their exact fp32 attention record (m, l, o) for the g query rows
// starts the running merge. Scores use the unrotated q and keys (a rotation
// leaves dot products unchanged); the value sum is rotated into the cache's
// domain when the cache is rotated. Whole CTA; sm: 64 KB of shared memory.
template <int CQ, typename T>
__device__ __forceinline__ void residual_record(const T* q, const T* res, int R, int g,
                                                const int8_t* signs, int hadamard, int part,
                                                float* sm, float* y, float* run_m, float* run_l,
                                                float (&acc)[kMaxHeads * (kD / CQ) / kThreads]) {
  constexpr int CW = kD / CQ;
  constexpr int PAIRS = kMaxHeads * CW / kThreads;
  const int tid = threadIdx.x;
  float* qf = sm;                                  // [g][128], scaled to log2 units
  float* kr = qf + kMaxHeads * kD;                 // [32][129]
  float* vr = kr + kTile * (kD + 1);               // [32][128]
  float* sc = vr + kTile * kD;                     // [g][32]
  const float qscale = kLog2e * kInvSqrt128;
  for (int n = 0; n < g; ++n) qf[n * kD + tid] = to_f32<T>(q[n * kD + tid]) * qscale;
  for (int t = 0; t < R; ++t) {
    kr[t * (kD + 1) + tid] = to_f32<T>(res[t * kD + tid]);
    vr[t * kD + tid] = to_f32<T>(res[(kTile + t) * kD + tid]);
  }
  __syncthreads();
  for (int idx = tid; idx < g * R; idx += kThreads) {
    const int n = idx / R, t = idx % R;
    float sdot = 0.0f;
    for (int c = 0; c < kD; ++c) sdot = __fmaf_rn(qf[n * kD + c], kr[t * (kD + 1) + c], sdot);
    sc[n * kTile + t] = sdot;
  }
  __syncthreads();
#pragma unroll
  for (int k = 0; k < PAIRS; ++k) {
    const int pi = tid + kThreads * k, n = pi / CW, c = pi % CW;
    if (n < g) {
      float m = -INFINITY;
      for (int t = 0; t < R; ++t) m = fmaxf(m, sc[n * kTile + t]);
      float l = 0.0f, o = 0.0f;
      for (int t = 0; t < R; ++t) {
        const float p = exp2f(sc[n * kTile + t] - m);
        l += p;
        o = __fmaf_rn(p, vr[t * kD + part * CW + c], o);
      }
      acc[k] = o;
      if (c == 0) {
        run_m[n] = m;
        run_l[n] = l;
      }
    }
  }
  if (CQ == 1 && hadamard) {                       // o R = FWHT(o * signs) / sqrt(128)
#pragma unroll
    for (int k = 0; k < PAIRS; ++k) {
      const int pi = tid + kThreads * k, c = pi % CW;
      if (pi / CW < g) y[pi] = (signs && signs[c] < 0) ? -acc[k] : acc[k];
    }
    __syncthreads();
    fwht_smem(y, g);
#pragma unroll
    for (int k = 0; k < PAIRS; ++k) {
      const int pi = tid + kThreads * k;
      if (pi / CW < g) acc[k] = y[pi] * kInvSqrt128;
    }
  }
  __syncthreads();
}

template <int CQ, typename T>
__global__ void __launch_bounds__(kThreads, 16) decode_merge_kernel(const float* partial, float* out,
                                                                const int8_t* signs,
                                                                uint32_t* status, int Hq, int H,
                                                                int g, int splits, int s_lo,
                                                                int u_lo, int hadamard,
                                                                const T* q, const T* residual,
                                                                int R, const int32_t* n_rows,
                                                                int cap, int msm_bytes) {
  // the next decode call's split grid may launch now (it waits for this grid
  // before writing the workspace)
  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
  // everything up to the wait reads only this call's inputs, so it overlaps
  // the split grid's tail
  bool row_ok = true;
  if (n_rows) {                  // a token count per batch row: its own residual tokens
    const int n = n_rows[blockIdx.x / H];
    row_ok = n >= 1 && n <= cap;
    R = row_ok ? n % kTile : 0;
    if (!row_ok && threadIdx.x == 0 && blockIdx.x % H == 0 && blockIdx.y == 0)
      set_status(status, RQ_STATUS_BAD_POSITION);
  }
  constexpr int CW = kD / CQ;          // channels of this CTA
  constexpr int CH = CW / 4;           // 16-byte pieces of a record's o slice
  constexpr int SLOT = CH + 1;         // pieces per (row, split): o slice, then (m, l, pad)
  constexpr int PAIRS = kMaxHeads * CW / kThreads;   // (row, channel) pairs per thread, at most
  static_assert(PAIRS >= 1, "every thread owns a (row, channel) pair");
  extern __shared__ float4 msm[];
  __shared__ float wgt[kMaxHeads][kMergeChunk];
  __shared__ float run_m[kMaxHeads], run_l[kMaxHeads], run_scale[kMaxHeads];
  __shared__ float y[kMaxHeads * kD];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int batch = blockIdx.x / H, h = blockIdx.x % H, part = blockIdx.y;
  const long long row0 = static_cast<long long>(batch) * Hq + h * g;
  const int rs = splits * kPart;                               // floats between query rows
  const int ns = static_cast<int>(blockIdx.x) < u_lo ? s_lo : splits;   // this unit's records
  const float* base = partial + row0 * rs;                     // row 0, split 0
  // sign flips of the thread's channels for the rotation back (bit k: pair k)
  uint32_t negmask = 0;
  if (CQ == 1 && hadamard && signs) {
#pragma unroll
    for (int k = 0; k < PAIRS; ++k)
      if (signs[(tid + kThreads * k) % CW] < 0) negmask |= 1u << k;
  }
  // splits per chunk: shared budget, and at most kMergeChunk (four weights per lane)
  const int cs_max = min(kMergeChunk, msm_bytes / (g * SLOT * 16));
  if (tid < kMaxHeads) {
    run_m[tid] = -INFINITY;
    run_l[tid] = 0.0f;
  }
  float acc[PAIRS];
#pragma unroll
  for (int k = 0; k < PAIRS; ++k) acc[k] = 0.0f;
  __syncthreads();
  if (R > 0)
    residual_record<CQ, T>(q + row0 * kD, residual + (static_cast<long long>(batch) * H + h) * 2 * kTile * kD,
                           R, g, signs, hadamard, part, reinterpret_cast<float*>(msm), y, run_m, run_l,
                           acc);
  const uint32_t sbase = static_cast<uint32_t>(__cvta_generic_to_shared(msm));
  asm volatile("griddepcontrol.wait;\n" ::: "memory");

  for (int c0 = 0; c0 < ns; c0 += cs_max) {
    const int cs = min(cs_max, ns - c0);
    // piece x = (n cs + sl) SLOT + i: i < CH the o slice, i == CH (m, l, pad,
    // pad); the thread steps x by kThreads with a mixed-radix carry instead
    // of dividing per piece
    const int npieces = g * cs * SLOT;
    {
      constexpr int DI = kThreads % SLOT, DR = kThreads / SLOT;
      int i = tid % SLOT, sl = tid / SLOT, n = sl / cs;
      sl -= n * cs;
      for (int x = tid; x < npieces; x += kThreads) {
        const int off = n * rs + (c0 + sl) * kPart + (i < CH ? part * CW + 4 * i : kD);
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(sbase + 16 * x), "l"(base + off));
        i += DI;
        sl += DR;
        if (i >= SLOT) {
          i -= SLOT;
          ++sl;
        }
        while (sl >= cs) {
          sl -= cs;
          ++n;
        }
      }
    }
    asm volatile("cp.async.commit_group;\n" ::);
    asm volatile("cp.async.wait_group 0;\n" ::);
    __syncthreads();
    // warp w: rows w, w + 4; lanes over the chunk's splits (four per lane)
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      const int n = warp + kWarps * k;
      if (n < g) {
        float mv[kMergeChunk / 32], lv[kMergeChunk / 32], mx = -INFINITY;
#pragma unroll
        for (int r = 0; r < kMergeChunk / 32; ++r) {
          const int sl = lane + 32 * r;
          mv[r] = -INFINITY;
          lv[r] = 0.0f;
          if (sl < cs) {
            const float4 ml = msm[(n * cs + sl) * SLOT + CH];
            mv[r] = ml.x;
            lv[r] = ml.y;
          }
          mx = fmaxf(mx, mv[r]);
        }
#pragma unroll
        for (int off = 16; off >= 1; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
        const float mold = run_m[n];
        const float mnew = fmaxf(mold, mx);
        float l = 0.0f;
#pragma unroll
        for (int r = 0; r < kMergeChunk / 32; ++r) {
          const int sl = lane + 32 * r;
          const float wv = (mv[r] == -INFINITY) ? 0.0f : exp2f(mv[r] - mnew);
          if (sl < cs) wgt[n][sl] = wv;
          l += wv * lv[r];
        }
#pragma unroll
        for (int off = 16; off >= 1; off >>= 1) l += __shfl_xor_sync(0xffffffffu, l, off);
        __syncwarp();
        if (lane == 0) {
          const float sc = (mold == -INFINITY) ? 0.0f : exp2f(mold - mnew);
          run_scale[n] = sc;
          run_l[n] = run_l[n] * sc + l;
          run_m[n] = mnew;
        }
      }
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < PAIRS; ++k) {
      const int pi = tid + kThreads * k, n = pi / CW, c = pi % CW;
      if (n < g) {
        float a = acc[k] * run_scale[n];
        const float* o = reinterpret_cast<const float*>(msm + n * cs * SLOT) + c;
        const float* wn = wgt[n];
#pragma unroll 4
        for (int sl = 0; sl < cs; ++sl) a += wn[sl] * o[sl * SLOT * 4];
        acc[k] = a;
      }
    }
    __syncthreads();
  }
#pragma unroll
  for (int k = 0; k < PAIRS; ++k) {
    const int n = (tid + kThreads * k) / CW;
    if (n < g) {
      const float L = run_l[n];
      float v = L > 0.0f ? acc[k] / L : 0.0f;
      if (row_ok && (!(L > 0.0f) || !isfinite(v))) {
        set_status(status, RQ_STATUS_NUMERIC);
        if (!isfinite(v)) v = 0.0f;
      }
      if (!row_ok) v = 0.0f;
      acc[k] = v;
    }
  }
  if (CQ == 1 && hadamard) {
    // FWHT of each row: thread c holds channel c of every row (acc[k] is row
    // k); strides 1 .. 16 are lane exchanges, strides 32 and 64 go through
    // shared memory. Every output is one fp32 a + b or a - b, as in the
    // butterfly order of the in-place transform.
#pragma unroll
    for (int st = 1; st <= 16; st <<= 1) {
      const bool up = lane & st;
#pragma unroll
      for (int k = 0; k < PAIRS; ++k) {
        const float o = __shfl_xor_sync(0xffffffffu, acc[k], st);
        acc[k] = up ? o - acc[k] : acc[k] + o;
      }
    }
#pragma unroll
    for (int st = 32; st <= 64; st <<= 1) {
      const bool up = tid & st;
#pragma unroll
      for (int k = 0; k < PAIRS; ++k)
        if (k < g) y[k * kD + tid] = acc[k];
      __syncthreads();
#pragma unroll
      for (int k = 0; k < PAIRS; ++k) {
        if (k < g) {
          const float o = y[k * kD + (tid ^ st)];
          acc[k] = up ? o - acc[k] : acc[k] + o;
        }
      }
      __syncthreads();
    }
#pragma unroll
    for (int k = 0; k < PAIRS; ++k) {
      const float v = acc[k] * kInvSqrt128;
      acc[k] = (negmask >> k) & 1u ? -v : v;
    }
  }
#pragma unroll
  for (int k = 0; k < PAIRS; ++k) {
    const int pi = tid + kThreads * k, n = pi / CW, c = pi % CW;
    if (n < g) out[(row0 + n) * kD + part * CW + c] = acc[k];
  }
}

// The merge's shared-memory records area for channel parts of 128 / cq: one
// round trip for every split of a unit when it fits (at most kMergeSmem), the
// residual record's 38 KB when rows may hold residual tokens.
inline int merge_smem_bytes(const DecodeArgs& a, int cq, bool residual) {
  const long long need = static_cast<long long>(a.g) * a.splits * (kD / cq / 4 + 1) * 16;
  const long long res = residual ? (kMaxHeads * kD + kTile * (kD + 1) + kTile * kD + kMaxHeads * kTile) * 4 : 0;
  return static_cast<int>(std::min<long long>(kMergeSmem, std::max(need, res)));
}

// split kernel, then the merge kernel as its programmatic dependent (it
// overlaps the split grid's tail and waits for it before reading); res_layer:
// this layer's residual windows (R > 0 tokens) or null
template <typename T>
inline rq_status launch_decode_t(DecodeArgs a, float* out, const void* res_layer, int R,
                                 cudaStream_t s) {
  int dev = 0, sms = 0, smem_sm = 0, reserved = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&reserved, cudaDevAttrReservedSharedMemoryPerBlock, dev) != cudaSuccess)
    return RQ_ERR_CUDA;
  const long long units = static_cast<long long>(a.B) * a.H;
  const long long nlo = static_cast<long long>(a.u_lo) * a.s_lo;
  const long long nsplit = nlo + (units - a.u_lo) * a.splits;
  // four groups per CTA when the query group takes the merged hi/lo MMA
  // (g <= 4: measured 2-3 % faster on those layers), one otherwise (g = 8:
  // 2-3 % slower as four groups)
  const int G = a.g <= kMaxHeads / 2 ? kGroups : 1;
  const bool residual = R > 0 || a.n_rows != nullptr;
  auto merge_kernel = [](int cq) {
    return cq == 1 ? decode_merge_kernel<1, T> : cq == 2 ? decode_merge_kernel<2, T>
                   : cq == 4 ? decode_merge_kernel<4, T> : decode_merge_kernel<8, T>;
  };
  // Merge CTAs beside the split CTAs: one fits on an SM (its <= 32
  // registers a thread take the 4,096 the 120-register split kernel leaves),
  // so the merge grid may have at most one CTA per SM. A whole row per CTA
  // for a rotated cache (the rotation mixes channels), else the most channel
  // parts (8, 4, 2) that keep units x parts within the SMs; and its shared
  // memory must fit in what the split CTAs of an SM leave.
  // Only for calls issued back to back (not a.mix): between other kernels
  // nothing overlaps the next call, and the 128-register kernel with the
  // merge grid starting where split CTAs have left was 3-7 % faster.
  int cq = a.hadamard ? 1 : 8;
  while (cq > 1 && units * cq > sms) cq >>= 1;
  int msm = merge_smem_bytes(a, cq, residual);
  bool co = units <= sms && !a.mix;
  if (co) {
    cudaFuncAttributes fa;
    if (cudaFuncGetAttributes(&fa, merge_kernel(cq)) != cudaSuccess) return RQ_ERR_CUDA;
    const int split_ctas = kGroups / G;                 // resident per SM
    const int left = smem_sm - split_ctas * (G * kGroupBytes + reserved);
    co = static_cast<int>(fa.sharedSizeBytes) + msm + reserved <= left;
  }
  if (!co) {
    // a whole row per CTA for a rotated cache, a quarter of the channels
    // otherwise (four times the CTAs), an eighth when there are few (batch,
    // kv head) units (the records of a unit are then many, and more CTAs
    // pull them in parallel)
    cq = a.hadamard ? 1 : (units <= 32 ? 8 : 4);
    msm = kMergeSmem;
  }
  a.early = (co || G == 1) ? 1 : 0;
  auto kern = co ? decode_split_kernel_co<T> : decode_split_kernel<T>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kSplitSmem) != cudaSuccess ||
      cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout,
                           cudaSharedmemCarveoutMaxShared) != cudaSuccess)
    return RQ_ERR_CUDA;
  // a programmatic dependent of whatever precedes it in the stream: it
  // launches early only after a grid that allows it (a decode merge), and
  // waits for that grid before writing
  cudaLaunchConfig_t scfg = {};
  scfg.gridDim = dim3(static_cast<unsigned>((nsplit + G - 1) / G));
  scfg.blockDim = dim3(kThreads * G);
  scfg.dynamicSmemBytes = G * kGroupBytes;
  scfg.stream = s;
  cudaLaunchAttribute sattr[1];
  sattr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  sattr[0].val.programmaticStreamSerializationAllowed = 1;
  scfg.attrs = sattr;
  scfg.numAttrs = 1;
  if (cudaLaunchKernelEx(&scfg, kern, a) != cudaSuccess) return RQ_ERR_CUDA;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(units), static_cast<unsigned>(cq));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = msm;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  auto mk = merge_kernel(cq);
  if (cudaFuncSetAttribute(mk, cudaFuncAttributeMaxDynamicSharedMemorySize, kMergeSmem) != cudaSuccess ||
      cudaFuncSetAttribute(mk, cudaFuncAttributePreferredSharedMemoryCarveout,
                           cudaSharedmemCarveoutMaxShared) != cudaSuccess)
    return RQ_ERR_CUDA;
  if (cudaLaunchKernelEx(&cfg, mk, static_cast<const float*>(a.partial), out, a.signs, a.status,
                         a.Hq, a.H, a.g, a.splits, a.s_lo, a.u_lo, a.hadamard, static_cast<const T*>(a.q),
                         static_cast<const T*>(res_layer), R, a.n_rows, a.nblk * kTile, msm) != cudaSuccess)
    return RQ_ERR_CUDA;
  return launch_status();
}

// Resident splits per SM on the current device: the smaller of the resident
// one-group CTAs and kGroups x the resident four-group CTAs (occupancy
// queries; both are 4 on GB300).
template <typename T>
inline rq_status split_ctas_per_sm_t(int* per_sm) {
  auto kern = decode_split_kernel<T>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kSplitSmem) != cudaSuccess ||
      cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout,
                           cudaSharedmemCarveoutMaxShared) != cudaSuccess)
    return RQ_ERR_CUDA;
  int v1 = 0, v4 = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v1, kern, kThreads, kGroupBytes) != cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v4, kern, kThreads * kGroups, kSplitSmem) != cudaSuccess)
    return RQ_ERR_CUDA;
  const int v = std::min(v1, v4 * kGroups);
  *per_sm = v > 0 ? v : 1;
  return RQ_OK;
}

}  // namespace dk

// one instance per input dtype, each in its own translation unit
// (decode_f16.cu, decode_bf16.cu) so that the two compile in parallel
rq_status launch_decode_f16(const dk::DecodeArgs& a, float* out, const void* res_layer, int R,
                            cudaStream_t s);
rq_status launch_decode_bf16(const dk::DecodeArgs& a, float* out, const void* res_layer, int R,
                             cudaStream_t s);
rq_status decode_split_ctas_per_sm(int* per_sm);

}  // namespace rq
