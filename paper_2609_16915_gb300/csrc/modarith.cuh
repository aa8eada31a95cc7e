// Word-level modular arithmetic for the NTT primes: the 28-bit set (16p <
// 2^32, so lazily reduced residues up to 8p still fit a 32-bit register) and
// the 31-bit set (2p < 2^32: residues below 2p).
//
// Residues are kept "lazy": a value congruent to the residue but possibly a
// few multiples of p above it.  Every function states the range it accepts
// and the range it returns.
#pragma once
#include <stdint.h>

namespace rosetta {

// Shoup multiplication by a constant w < p with companion ws = floor(w 2^32 / p):
// for any 32-bit y returns y*w mod p as a value in [0, 2p).
__device__ __forceinline__ uint32_t shoup_mul(uint32_t y, uint32_t w, uint32_t ws, uint32_t p) {
  const uint32_t q = __umulhi(y, ws);
  return y * w - q * p;
}

// Montgomery reduction with R = 2^32, p_inv = p^{-1} mod 2^32.
// For T < p * 2^32 returns a value in (0, 2p) congruent to T * 2^-32 mod p.
// The low words of T and m*p agree, so (T - m p) / 2^32 = hi(T) - hi(m p).
__device__ __forceinline__ uint32_t redc(uint64_t T, uint32_t p, uint32_t p_inv) {
  const uint32_t m = static_cast<uint32_t>(T) * p_inv;
  const uint32_t t = __umulhi(m, p);
  return static_cast<uint32_t>(T >> 32) - t + p;
}

// Quotient of the explicit CRT, round(sum_q y_q / p_q), from ysum = sum_q
// (y_q >> 2) with every y_q < 8 p_q.  The primes lie in (2^28 - 2^18, 2^28),
// so y / 2^28 undershoots y / p by less than 8 (2^28 - p) / 2^28 < 2^-7 per
// prime (the shift adds under 2^-26); the four together by less than 2^-5.
// The exact sum is an integer plus X / M with |X| <= 2^110 < M / 3.99 (the
// bound every accepted parameter set meets), so the estimate stays within
// 0.29 of that integer and rounds to it.
__device__ __forceinline__ uint32_t crt_quotient(uint32_t ysum) { return (ysum + (1u << 25)) >> 26; }

// The same for the three primes in (2^31 - 2^19, 2^31), from ysum = sum_q
// (y_q >> 3) with every y_q < 2 p_q < 2^32 (the sum stays below 2^31).
// y / 2^31 undershoots y / p by less than 2 (2^31 - p) / 2^31 < 2^-11 per
// prime (the shift adds under 2^-28); the three together by less than 2^-9.
// Only parameter sets whose exact integer value X obeys |X| <= 0.45 M take
// this prime set, so the estimate stays within 0.46 of the integer.
__device__ __forceinline__ uint32_t crt_quotient31(uint32_t ysum) { return (ysum + (1u << 27)) >> 28; }

// x in [0, 2b) -> [0, b) for a bound b: one subtraction when x >= b.
__device__ __forceinline__ uint32_t cond_sub(uint32_t x, uint32_t b) {
  return min(x, x - b);
}

}  // namespace rosetta
