// Conversion of the raw bootstrapping key to the transform domain the
// external product uses: for every GGSW row polynomial and every NTT prime,
// the centred words (value - 2^64 when >= 2^63) reduced mod p, forward
// negacyclic NTT (bit-reversed order, the order the blind-rotation kernel's
// forward transforms produce), fully reduced and scaled by 2^32 crt_c mod p:
// 2^32 is the Montgomery form (the kernel's Montgomery reduction of digit x
// key products returns the plain product), crt_c = N^-1 (M/p)^-1 the factor
// the explicit CRT needs after the inverse transform, applied here once per
// key word instead of once per output coefficient and step (the inverse
// transform is linear).
//
// Output layout [i][prime][row][component][N] uint32, so that one CTA of the
// blind-rotation (or trace) kernel streams one contiguous block per step.
// The same conversion serves the trace's automorphism keys.  Either prime
// set: the four 28-bit primes (lazy transforms) or the three 31-bit primes
// of the three-prime blind rotation (P31 transforms); gridDim.y is the number
// of primes.
#include "internal.h"
#include "ntt.cuh"

namespace rosetta {

template <int LOGN, bool P31>
__global__ void __launch_bounds__((1 << LOGN) / 8)
    bsk_transform_kernel(const uint64_t *__restrict__ raw, uint32_t *__restrict__ out, const uint2 *__restrict__ tw_all,
                         const CrtConsts cc, uint32_t rows) {
  using S = NttShape<LOGN, 8>;
  constexpr uint32_t N = S::N, T = S::T;
  extern __shared__ __align__(16) unsigned char smem[];
  uint2 *tw = reinterpret_cast<uint2 *>(smem);
  uint32_t *xb = reinterpret_cast<uint32_t *>(tw + N);
  const uint32_t tau = threadIdx.x;
  const uint32_t poly = blockIdx.x;  // (i * rows + r) * 2 + c over the raw layout
  const uint32_t q = blockIdx.y;
  const PrimeConsts pc = cc.pr[q];
  const uint32_t p = pc.p;
  for (uint32_t m = tau; m < N; m += T) tw[m] = tw_all[q * N + m];

  const uint64_t *src = raw + static_cast<size_t>(poly) * N;
  uint32_t x[1][8];
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    const uint64_t w = src[tau + e * T];
    const bool neg = static_cast<int64_t>(w) < 0;
    const uint64_t mag = neg ? 0ull - w : w;
    const uint32_t r = static_cast<uint32_t>(mag % p);
    x[0][e] = (neg && r) ? p - r : r;
  }
  __syncthreads();
  ntt_forward<LOGN, 8, 1, 1, P31>(x, tw, xb, tau, p);

  const uint32_t c = poly % 2;
  const uint32_t r = (poly / 2) % rows;
  const uint32_t i = poly / (2 * rows);
  uint32_t *dst = out + (((static_cast<size_t>(i) * gridDim.y + q) * rows + r) * 2 + c) * N + 8 * tau;
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    uint32_t v = P31 ? cond_sub(x[0][e], p)                                                      // < 2p -> < p
                     : cond_sub(cond_sub(cond_sub(cond_sub(x[0][e], 8 * p), 4 * p), 2 * p), p);  // < 16p -> < p
    v = cond_sub(shoup_mul(v, pc.key_scale, pc.key_scale_s, p), p);
    dst[e] = v;
  }
}

template <int LOGN, bool P31>
static cudaError_t launch_key_t(const uint64_t *raw, uint32_t *out, const uint2 *tw, const CrtConsts &cc,
                                uint32_t count, uint32_t rows, cudaStream_t s) {
  using S = NttShape<LOGN, 8>;
  const size_t smem = S::N * sizeof(uint2) + S::XB_WORDS * sizeof(uint32_t);
  auto kern = bsk_transform_kernel<LOGN, P31>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  dim3 grid(count * rows * 2, P31 ? kPrimes31 : kPrimes, 1);
  kern<<<grid, S::T, smem, s>>>(raw, out, tw, cc, rows);
  return cudaGetLastError();
}

template <bool P31>
static cudaError_t launch_key_n(const uint64_t *raw, uint32_t *out, const uint2 *tw, const CrtConsts &cc,
                                uint32_t logN, uint32_t count, uint32_t rows, cudaStream_t s) {
  switch (logN) {
    case 8: return launch_key_t<8, P31>(raw, out, tw, cc, count, rows, s);
    case 9: return launch_key_t<9, P31>(raw, out, tw, cc, count, rows, s);
    case 10: return launch_key_t<10, P31>(raw, out, tw, cc, count, rows, s);
    case 11: return launch_key_t<11, P31>(raw, out, tw, cc, count, rows, s);
    case 12: return launch_key_t<12, P31>(raw, out, tw, cc, count, rows, s);
    case 13: return launch_key_t<13, P31>(raw, out, tw, cc, count, rows, s);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_key_transform(const uint64_t *raw, uint32_t *out, const uint2 *tw, const CrtConsts &cc,
                                 uint32_t logN, uint32_t count, uint32_t rows, cudaStream_t s, uint32_t primes) {
  if (primes == kPrimes) return launch_key_n<false>(raw, out, tw, cc, logN, count, rows, s);
  if (primes == kPrimes31) return launch_key_n<true>(raw, out, tw, cc, logN, count, rows, s);
  return cudaErrorInvalidValue;
}

// The bootstrapping key: n GGSWs of (k+1) l = 2 l rows each.
cudaError_t launch_bsk_transform(const uint64_t *raw, uint32_t *out, const uint2 *tw, const CrtConsts &cc,
                                 uint32_t logN, uint32_t n, uint32_t level, uint32_t primes, cudaStream_t s) {
  return launch_key_transform(raw, out, tw, cc, logN, n, 2 * level, s, primes);
}

}  // namespace rosetta
