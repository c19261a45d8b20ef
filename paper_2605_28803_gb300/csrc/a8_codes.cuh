// Encodings of 8-bit activation codes for the W4A8 GEMM (device helpers).
//
// A code q in [-127, 127] enters the tensor cores as u = q + 128 = 16 hi + lo, split into two
// E4M3 operand planes against the same int4 weight operand (w + 8) 2^-9: the high nibble as
// the E4M3 value hi 2^-5 (a normal number for hi >= 1) and the low nibble as lo 2^-9 (the E4M3
// byte equal to lo: subnormal below 8, normal from 8).  Both products are exact multiples of
// 2^-18, and sum_k u (w + 8) 2^-18 is the FP32 accumulator, exact while it stays below 2^24
// units (255 x 15 x K < 2^24, i.e. K <= 4386).
#pragma once

#include <cstdint>

namespace qvla {

// E4M3 bytes of v 2^-5 for the four bytes v in [0, 15] of a word: 0x00 0x10 0x18 0x1C 0x20
// 0x22 0x24 0x26 for v = 0..7, v + 32 for v >= 8.
__device__ __forceinline__ uint32_t hi_plane_bytes(uint32_t v) {
  const uint32_t t = v & 0x07070707u;
  const uint32_t x = t | (t >> 4);
  const uint32_t sel = (x & 0xFFu) | ((x >> 8) & 0xFF00u);  // the four 3-bit indices as nibbles
  const uint32_t small = __byte_perm(0x1C181000u, 0x26242220u, sel);
  const uint32_t big = (v & 0x08080808u) >> 3;  // 1 where v >= 8
  const uint32_t mask = big * 0xFFu;
  return (small & ~mask) | ((v | 0x20202020u) & mask);
}

// The plane words of 4 even-k and 4 odd-k codes (two's-complement bytes e and o): high plane
// (he, ho) and low plane (le, lo).  The GEMM stores each group of 8 as k0 k2 k4 k6 k1 k3 k5 k7,
// i.e. the even word, then the odd word.
__device__ __forceinline__ void a8_planes(uint32_t e, uint32_t o, uint32_t& he, uint32_t& ho, uint32_t& le,
                                          uint32_t& lo) {
  const uint32_t e8 = e ^ 0x80808080u, o8 = o ^ 0x80808080u;  // bytes of q + 128
  le = e8 & 0x0F0F0F0Fu;
  lo = o8 & 0x0F0F0F0Fu;
  he = hi_plane_bytes((e8 >> 4) & 0x0F0F0F0Fu);
  ho = hi_plane_bytes((o8 >> 4) & 0x0F0F0F0Fu);
}

}  // namespace qvla
