// dard_rope.cuh - rotary position embedding (RoPE) of the augmented sequence, device side.
//
// Row positions follow Sec. 3.1 of arXiv 2608.26574: x^i and its shadow copy s^i share the
// positional embedding of position i, so original row r of a sequence sits at position r
// and shadow row N + k at position shadow_src[k]. The rotation itself is RoPE (Su et al.,
// RoFormer, 2021): the pair (a, b) at frequency index i of a row at position p becomes
// (a cos(p f_i) - b sin(p f_i), a sin(p f_i) + b cos(p f_i)), f_i = theta^(-2i/D), with
// pairs (2i, 2i + 1) (DARD_ROPE_INTERLEAVED) or (i, i + D/2) (DARD_ROPE_HALF).
//
// Angle arithmetic: f_i arrives as a float and the float of its remainder, so p f_i is
// formed as an unevaluated sum of two floats (the rounding error of p * f_hi recovered
// exactly by an FMA). The reduction modulo 2 pi is the additive two-constant (Cody-Waite)
// method: k = rint(a / 2 pi), r = (a - k C1) - k C2 with C1 = fl(2 pi) and
// C2 = fl(2 pi - C1). With |p| <= 2^20 and f_i <= 1, a - k C1 is exact (it is a multiple
// of 2^-22 below 4 in magnitude), so r carries two roundings of about 1.2e-7 each;
// cos and sin then come from the hardware approximations, whose documented absolute error
// on [-pi, pi] is below 2^-21.
#pragma once
#include <cuda_bf16.h>

#include "dard_internal.h"

namespace dard {

constexpr float kTwoPiHi = 6.2831854820251465f;        // fl(2 pi)
constexpr float kTwoPiLo = -1.7484555314695172e-07f;   // fl(2 pi - kTwoPiHi)
constexpr float kInvTwoPi = 0.15915493667125702f;      // fl(1 / (2 pi))

// cos and sin of pos * (f_hi + f_lo).
__device__ __forceinline__ void rope_cos_sin(int pos, float f_hi, float f_lo, float& c,
                                             float& s) {
  const float x = static_cast<float>(pos);  // exact: |pos| <= 2^20
  const float a_hi = x * f_hi;
  const float a_lo = fmaf(x, f_hi, -a_hi) + x * f_lo;
  const float k = rintf(a_hi * kInvTwoPi);
  float r = fmaf(-k, kTwoPiHi, a_hi);
  r = fmaf(-k, kTwoPiLo, r);
  r += a_lo;
  __sincosf(r, &s, &c);
}

// Position of sequence-relative row r (Sec. 3.1: the shadow copy of position j sits at j).
__device__ __forceinline__ int rope_position(const AttnParams& p, const SeqDesc& sd, int r) {
  return r < sd.n_orig ? r : __ldg(p.shadow_src + sd.sh_off + (r - sd.n_orig));
}

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }
__device__ __forceinline__ uint32_t bf_pack(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}

// An interleaved pair held in one bf16x2 word: (a, b) -> (a c - b s, a s + b c).
__device__ __forceinline__ uint32_t rope_pair_word(uint32_t w, float c, float s) {
  const float a = bf_lo(w), b = bf_hi(w);
  return bf_pack(fmaf(a, c, -b * s), fmaf(a, s, b * c));
}

// Sixteen bytes of a bf16 row (elements 8 j .. 8 j + 7, four interleaved pairs) at
// position pos; f points at the (hi, lo) pairs of frequencies 4 j .. 4 j + 3.
__device__ __forceinline__ void rope_chunk_interleaved(uint4& u, int pos, const float* f) {
  float c, s;
  rope_cos_sin(pos, f[0], f[1], c, s);
  u.x = rope_pair_word(u.x, c, s);
  rope_cos_sin(pos, f[2], f[3], c, s);
  u.y = rope_pair_word(u.y, c, s);
  rope_cos_sin(pos, f[4], f[5], c, s);
  u.z = rope_pair_word(u.z, c, s);
  rope_cos_sin(pos, f[6], f[7], c, s);
  u.w = rope_pair_word(u.w, c, s);
}

// Half pairing: a word of the first half (a0, a1) and the word D/2 elements later (b0, b1)
// form pairs (a0, b0) and (a1, b1). Returns this side's rotated word: the first half takes
// a c - b s, the second a s + b c.
__device__ __forceinline__ uint32_t rope_half_word(uint32_t own, uint32_t other, bool own_first,
                                                   float c0, float s0, float c1, float s1) {
  const float o0 = bf_lo(own), o1 = bf_hi(own), t0 = bf_lo(other), t1 = bf_hi(other);
  if (own_first) return bf_pack(fmaf(o0, c0, -t0 * s0), fmaf(o1, c1, -t1 * s1));
  return bf_pack(fmaf(t0, s0, o0 * c0), fmaf(t1, s1, o1 * c1));
}

// Sixteen bytes of a bf16 row in the half pairing: `own` holds elements e .. e + 7 of one
// half, `other` the same offsets of the other half; f points at the (hi, lo) pairs of the
// eight frequencies e' .. e' + 7 (e' = e mod D/2). Rotates `own` only.
__device__ __forceinline__ void rope_chunk_half(uint4& own, const uint4& other, bool own_first,
                                                int pos, const float* f) {
  float c0, s0, c1, s1;
  rope_cos_sin(pos, f[0], f[1], c0, s0);
  rope_cos_sin(pos, f[2], f[3], c1, s1);
  own.x = rope_half_word(own.x, other.x, own_first, c0, s0, c1, s1);
  rope_cos_sin(pos, f[4], f[5], c0, s0);
  rope_cos_sin(pos, f[6], f[7], c1, s1);
  own.y = rope_half_word(own.y, other.y, own_first, c0, s0, c1, s1);
  rope_cos_sin(pos, f[8], f[9], c0, s0);
  rope_cos_sin(pos, f[10], f[11], c1, s1);
  own.z = rope_half_word(own.z, other.z, own_first, c0, s0, c1, s1);
  rope_cos_sin(pos, f[12], f[13], c0, s0);
  rope_cos_sin(pos, f[14], f[15], c1, s1);
  own.w = rope_half_word(own.w, other.w, own_first, c0, s0, c1, s1);
}

// 16-byte chunk c (elements 8 c .. 8 c + 7) of row `row` in a 128-row tile stored as 64-column
// blocks of 128 rows x 128 bytes with the 128-byte swizzle (chunk index XOR row % 8), the
// layout the TMA loads and the MMA descriptors use.
__device__ __forceinline__ uint4* sw128_chunk(uint8_t* tile, int row, int c) {
  return reinterpret_cast<uint4*>(tile + (c >> 3) * (128 * 128) + row * 128 +
                                  (((c & 7) ^ (row & 7)) << 4));
}

// Rotates row `row` of a bf16 query tile in shared memory (layout of sw128_chunk) in place.
template <int D>
__device__ __forceinline__ void rope_tile_row(const AttnParams& p, uint8_t* tile, int row,
                                              int pos) {
  if (p.rope_style == DARD_ROPE_INTERLEAVED) {
#pragma unroll 4
    for (int c = 0; c < D / 8; ++c) {
      uint4* ptr = sw128_chunk(tile, row, c);
      uint4 u = *ptr;
      rope_chunk_interleaved(u, pos, p.rope_f + 8 * c);
      *ptr = u;
    }
  } else {
#pragma unroll 2
    for (int c = 0; c < D / 16; ++c) {
      uint4* pa = sw128_chunk(tile, row, c);
      uint4* pb = sw128_chunk(tile, row, c + D / 16);
      uint4 a = *pa, b = *pb;
      const uint4 a0 = a;
      rope_chunk_half(a, b, true, pos, p.rope_f + 16 * c);
      rope_chunk_half(b, a0, false, pos, p.rope_f + 16 * c);
      *pa = a;
      *pb = b;
    }
  }
}

}  // namespace dard
