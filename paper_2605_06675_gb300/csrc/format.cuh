// Packed block format: where each code of a 32-token x 128-channel block
// lives, shared by the quantizer (which writes it) and the decoder (which
// reads it). Storage is this library's own choice; the paper fixes only that
// per-head widths come from a static table (App. M, App. U).
//
// A block image is 128*b code words then 128 meta words. Lane L = 4 gid + tig
// (gid 0..7, tig 0..3) owns 4*b words of it: lane word w sits at block word
// 128 (w / 4) + 4 L + (w % 4). The lane's codes form 4 units u of 16
// registers psi = 4 x + y (class x, member y, both 0..3); a register holds two
// codes, half h = 0 / 1, which are the two fp16 halves of one MMA A-fragment
// register:
//   K, per-channel groups:  token 8 y + gid,        channel 32 u + 8 tig + 2 x + h
//   K, per-token groups:    token 8 x + gid,        channel 32 u + 8 tig + 2 y + h
//   V, either grouping:     token 8 y + 2 tig + h,  channel 32 u + 4 gid + x
// Unit u owns lane words b u .. b u + b - 1 ("unit words"). A 16-bit half has
// n = 16 / b slots; slot (w, k) puts the half-h code at bits 16 h + b k of
// unit word w. Widths that leave spare bits (b = 3, 5, 6, 7) chain the spare
// bits of the unit words, per half, into a spare stream that holds the
// leftover registers' codes, b bits each.
//
// Both halves of a register sit at the same offset, so one AND of a
// (shifted) unit word yields the pair as two fp16 subnormals c * 2^(E - 24):
// exact, ready for the tensor cores. E depends only on the class x (the
// decoder folds 2^-E into the other MMA operand or the output row).
#pragma once

#include <cstdint>

namespace rq {
namespace fmt {

__host__ __device__ constexpr int slots(int b) { return 16 / b; }
__host__ __device__ constexpr int spare(int b) { return 16 - b * (16 / b); }

// Location of register (x, y): leftover index `left` (>= 0), or main slot
// (w, k) when left < 0.
struct Loc {
  int left, w, k;
};

__host__ __device__ constexpr Loc location(int b, int x, int y) {
  if (b == 1 || b == 2 || b == 4 || b == 8) {
    const int n = 16 / b, s = x + 4 * y;
    return Loc{-1, s / n, s % n};
  }
  if (b == 3) {
    // x = 0: (0,0) (1,0) (2,0) left0; x = 1: (0,1) (1,1) (2,1) (1,4);
    // x = 2: (0,2) (1,2) (2,2) (2,4); x = 3: (0,3) (1,3) (2,3) (0,4)
    if (y < 3) return Loc{-1, y, x};
    return x == 0 ? Loc{0, 0, 0} : x == 1 ? Loc{-1, 1, 4} : x == 2 ? Loc{-1, 2, 4} : Loc{-1, 0, 4};
  }
  if (b == 5) {
    // x = 0: (y,0); x = 1: (y,1); x = 2: (4,0) (0,2) (1,2) left0;
    // x = 3: (4,1) (2,2) (3,2) (4,2)
    if (x < 2) return Loc{-1, y, x};
    if (x == 2) return y == 0 ? Loc{-1, 4, 0} : y == 3 ? Loc{0, 0, 0} : Loc{-1, y - 1, 2};
    return y == 0 ? Loc{-1, 4, 1} : Loc{-1, y + 1, 2};
  }
  const int psi = 4 * x + y, main = b == 6 ? 12 : 14;
  return psi < main ? Loc{-1, psi / 2, psi % 2} : Loc{psi - main, 0, 0};
}

// exponent of the extracted pair: the code sits at bit E of each half
__host__ __device__ constexpr int exponent(int b, int x) {
  return b == 1 ? x
       : b == 2 ? 2 * x
       : b == 3 ? (x == 1 ? 3 : x == 2 ? 6 : 0)
       : b == 4 ? 4 * (x & 1)
       : b == 5 ? 5 * (x & 1)
       : 0;
}

__host__ __device__ constexpr uint32_t pair_mask(int bits, int at) {
  return ((1u << bits) - 1u) * (0x00010001u << at);
}

// ---------------------------------------------------------------- writer ----
// OR the code pair P = c0 | c1 << 16 of register (x, y) into the unit words.
template <int B>
__device__ __forceinline__ void place(uint32_t (&uw)[B], int x, int y, uint32_t P) {
  const Loc l = location(B, x, y);
  if (l.left < 0) {
    // the slot's bits are still zero, so adding the shifted pair sets them
    // (one multiply-add instead of a shift and an OR)
    uw[l.w] += P * (1u << (B * l.k));
  } else if constexpr (spare(B) > 0) {
    constexpr int n = 16 / B, r = spare(B);
#pragma unroll
    for (int k = 0; k < B; ++k) {
      const int i = B * l.left + k;                 // spare-stream bit
      if (k == 0 || i % r == 0) {                   // a run of bits in one word starts
        const int len = (r - i % r) < (B - k) ? (r - i % r) : (B - k);
        uw[i / r] |= ((P >> k) & pair_mask(len, 0)) << (B * n + i % r);
      }
    }
  }
}

// ---------------------------------------------------------------- reader ----
// Register (x, y) of a unit as two fp16 subnormals c * 2^(E - 24),
// E = exponent(B, x).
template <int B>
__device__ __forceinline__ uint32_t extract(const uint32_t* uw, int x, int y) {
  const Loc l = location(B, x, y);
  if (l.left < 0) {
    if (B == 8) {
      return l.k == 0 ? (uw[l.w] & 0x00FF00FFu) : __byte_perm(uw[l.w], 0u, 0x4341u);
    }
    const int E = exponent(B, x);
    const int sh = B * l.k - E;
    return (uw[l.w] >> sh) & pair_mask(B, E);
  }
  uint32_t v = 0;
  if constexpr (spare(B) > 0) {
  constexpr int n = 16 / B, r = spare(B);
#pragma unroll
  for (int k = 0; k < B; ++k) {
    const int i = B * l.left + k;
    if (k == 0 || i % r == 0) {                        // a run of bits in one word starts
      const int len = (r - i % r) < (B - k) ? (r - i % r) : (B - k);
      v |= (uw[i / r] >> (B * n + i % r - k)) & pair_mask(len, k);
    }
  }
  }
  return v;
}

}  // namespace fmt
}  // namespace rq
