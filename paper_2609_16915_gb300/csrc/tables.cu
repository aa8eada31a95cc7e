// Host-side precomputation: twiddle tables and CRT constants for a set of NTT
// primes (the four 28-bit primes, or the three 31-bit ones).  Runs once per
// context and set.
#include <vector>

#include "internal.h"

namespace rosetta {
namespace {

using u128 = unsigned __int128;

uint32_t powmod(uint64_t b, uint64_t e, uint32_t p) {
  uint64_t r = 1;
  b %= p;
  while (e) {
    if (e & 1) r = r * b % p;
    b = b * b % p;
    e >>= 1;
  }
  return static_cast<uint32_t>(r);
}

bool is_prime(uint32_t p) {
  if (p < 2) return false;
  for (uint32_t d = 2; (uint64_t)d * d <= p; ++d)
    if (p % d == 0) return false;
  return true;
}

// Smallest generator of Z_p^*: g^((p-1)/f) != 1 for every prime factor f.
uint32_t generator(uint32_t p) {
  std::vector<uint32_t> fac;
  uint32_t m = p - 1;
  for (uint32_t d = 2; (uint64_t)d * d <= m; ++d) {
    if (m % d == 0) {
      fac.push_back(d);
      while (m % d == 0) m /= d;
    }
  }
  if (m > 1) fac.push_back(m);
  for (uint32_t g = 2; g < p; ++g) {
    bool ok = true;
    for (uint32_t f : fac)
      if (powmod(g, (p - 1) / f, p) == 1) {
        ok = false;
        break;
      }
    if (ok) return g;
  }
  return 0;
}

uint32_t bitrev(uint32_t x, uint32_t bits) {
  uint32_t r = 0;
  for (uint32_t i = 0; i < bits; ++i) r |= ((x >> i) & 1u) << (bits - 1 - i);
  return r;
}

uint32_t shoup(uint32_t w, uint32_t p) { return static_cast<uint32_t>((static_cast<uint64_t>(w) << 32) / p); }

}  // namespace

bool build_tables(uint32_t logN, uint32_t primes, uint2 *tw_host, CrtConsts *cc) {
  const uint32_t N = 1u << logN;
  if (primes != kPrimes && primes != kPrimes31) return false;
  const uint32_t *list = primes == kPrimes ? kPrimeList : kPrime31List;
  // 28-bit set in (2^28 - 2^18, 2^28): lazy residues up to 16p fit 32 bits and
  // the CRT quotient may use 2^28 in place of p; 31-bit set in
  // (2^31 - 2^19, 2^31): residues below 2p fit, the quotient uses 2^31
  const uint32_t top = primes == kPrimes ? 28 : 31, gap = primes == kPrimes ? 18 : 19;
  *cc = CrtConsts{};
  u128 M = 1;
  for (uint32_t q = 0; q < primes; ++q) M *= list[q];
  cc->M_mod64 = static_cast<uint64_t>(M);
  for (uint32_t q = 0; q < primes; ++q) {
    const uint32_t p = list[q];
    if (!is_prime(p) || (p - 1) % (2 * N) != 0 || p >= (1u << top) || p <= (1u << top) - (1u << gap)) return false;
    const uint32_t g = generator(p);
    if (!g) return false;
    const uint32_t psi = powmod(g, (p - 1) / (2 * N), p);  // primitive 2N-th root of unity
    if (powmod(psi, N, p) != p - 1) return false;
    for (uint32_t m = 0; m < N; ++m) {
      const uint32_t w = powmod(psi, bitrev(m, logN), p);
      tw_host[(size_t)q * N + m] = make_uint2(w, shoup(w, p));
    }
    PrimeConsts &pc = cc->pr[q];
    pc.p = p;
    uint32_t inv = 1;  // Newton iteration for p^{-1} mod 2^32
    for (int it = 0; it < 5; ++it) inv *= 2u - p * inv;
    pc.p_inv = inv;
    const u128 Mq = M / p;
    const uint32_t Mq_mod_p = static_cast<uint32_t>(Mq % p);
    const uint32_t Mq_inv = powmod(Mq_mod_p, p - 2, p);
    const uint32_t N_inv = powmod(N, p - 2, p);
    pc.crt_c = static_cast<uint32_t>(static_cast<uint64_t>(Mq_inv) * N_inv % p);
    pc.crt_cs = shoup(pc.crt_c, p);
    const uint64_t r_mont = (static_cast<uint64_t>(1) << 32) % p;
    pc.key_scale = static_cast<uint32_t>(r_mont * pc.crt_c % p);
    pc.key_scale_s = shoup(pc.key_scale, p);
    pc.Mp_mod64 = static_cast<uint64_t>(Mq);
  }
  return true;
}

}  // namespace rosetta
