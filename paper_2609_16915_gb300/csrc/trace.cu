// RLWE trace of a batch of GLWE ciphertexts (k = 1), one 4-CTA cluster per
// ciphertext.
//
// The paper isolates the constant coefficient of an RLWE ciphertext with a
// trace: a logarithmic sequence of Galois automorphisms and additions under
// which every other coefficient cancels (Background, "Scheme Conversion and
// Other Primitives", RLWE Trace Computation; used after each blind rotation
// of the Cryptographic Lookup Protocol).  Step s (s = 0 .. log2 N - 1) uses
// the automorphism X -> X^k, k = 2^(log2 N - s) + 1:
//     c <- c + KS_s(sigma_k(c)),  KS_s(A', B') = (0, B') - sum_l D_l(A') * key_s[l]
// where key_s[l] encrypts sigma_k(S) 2^(64 - l beta) under S.  After all steps
// the phase is N times the input's constant coefficient (N has no inverse on
// the torus Z_{2^64}; the factor stays).
//
// The products sum_l D_l * key_s[l][c] are computed exactly with the same
// four-prime NTT + explicit CRT machinery as blind rotation, split the same
// way: CTA r of the cluster transforms for prime r and owns coefficients
// [rN/4, (r+1)N/4).  Per step:
//   1. owners gather sigma_k(A), sigma_k(B) for their quarter (distributed
//      shared memory), write the digits of sigma_k(A) and keep sigma_k(B);
//   2. prime-CTAs transform digit pairs, multiply by key_s, inverse-transform
//      and send CRT-scaled residues to the owners;
//   3. owners: A -= X_0, B += sigma_k(B) - X_1.
//
// The same kernel in its plaintext-multiply mode computes, in one step,
// (P * A, P * B + Q) for a plaintext polynomial P (small signed
// coefficients) and Q: the ciphertext components are split into exact gadget
// digits (base_log * levels = 64) and multiplied by the rows P 2^(64 - l base_log)
// of a noiseless "key", which gives P * C exactly; this is the linear mapping
// a_s(X) [[x]] + b_s(X) of the lookup protocol (Cryptographic Lookup Protocol,
// Steps 2 and 3).
#include <cooperative_groups.h>

#include "dsmem.cuh"
#include "internal.h"
#include "ntt.cuh"

namespace rosetta {
namespace cg = cooperative_groups;

template <int LOGN>
struct TrShape {
  static constexpr int N = 1 << LOGN;
  static constexpr int E = 8;
  static constexpr int T = N / E;
  static constexpr int Q = N / 4;
  static constexpr int ITEMS = 2 * Q / T;  // 2 mask items then 2 body items per thread
  static constexpr int QE = E / 4;
};

template <int LOGN, bool PTMUL>
__global__ void __launch_bounds__(TrShape<LOGN>::T) trace_kernel(const TraceArgs a) {
  using B = TrShape<LOGN>;
  constexpr uint32_t N = B::N, T = B::T, Q = B::Q;
  constexpr uint32_t TWO_N = 2 * N;
  constexpr int E = B::E, ITEMS = B::ITEMS, QE = B::QE;

  cg::cluster_group cluster = cg::this_cluster();
  const uint32_t rank = cluster.block_rank();
  const uint32_t ct = blockIdx.x / 4;
  const uint32_t tau = threadIdx.x;

  extern __shared__ __align__(16) unsigned char smem[];
  uint2 *tw = reinterpret_cast<uint2 *>(smem);                  // [N]
  uint64_t *acc = reinterpret_cast<uint64_t *>(tw + N);         // [2][Q]
  uint64_t *sig_b = acc + 2 * Q;                                 // [Q] sigma_k(B) of the owned quarter
  uint32_t *res = reinterpret_cast<uint32_t *>(sig_b + Q);      // [4 primes][2][Q]
  uint32_t *xb = res + kPrimes * 2 * Q;                         // [XB_WORDS]
  int32_t *dig = reinterpret_cast<int32_t *>(xb + NttShape<LOGN, E>::XB_WORDS);  // [level][Q]

  const uint32_t p = a.cc.pr[rank].p;
  const uint32_t p_inv = a.cc.pr[rank].p_inv;

  for (uint32_t m = tau; m < N; m += T) tw[m] = a.tw[rank * N + m];
  const uint64_t *gin = a.glwe_in + static_cast<size_t>(ct) * 2 * N;
#pragma unroll
  for (int m = 0; m < ITEMS; ++m) {
    const uint32_t item = tau + m * T;
    const uint32_t c = item / Q, jl = item % Q;
    acc[c * Q + jl] = gin[c * N + rank * Q + jl];
  }
  cluster.sync();

  const uint32_t acc_s = smem_addr(acc), dig_s = smem_addr(dig), res_s = smem_addr(res);
  const uint32_t bits = a.base_log * (PTMUL ? a.level / 2 : a.level);
  const uint64_t Bmask = (1ull << a.base_log) - 1;
  const uint64_t Bhalf = 1ull << (a.base_log - 1);
  const uint64_t round_add = bits >= 64 ? 0 : (1ull << (63 - bits));
  const uint32_t round_sh = bits >= 64 ? 0 : 64 - bits;

  // multiply mode: level key rows = 2 x gadget levels (component-major)
  const uint32_t dlev = PTMUL ? a.level / 2 : a.level;
  constexpr uint32_t STEPS = PTMUL ? 1 : LOGN;
  for (uint32_t s = 0; s < STEPS; ++s) {
    const uint32_t k = PTMUL ? 1u : (1u << (LOGN - s)) + 1u;
    uint32_t kinv = k;  // k^{-1} mod 2^32 (Newton), hence mod 2N
#pragma unroll
    for (int it = 0; it < 5; ++it) kinv *= 2u - k * kinv;

    // ---- phase 1: gather sigma_k(c) for the owned quarter ----
    // coefficient j of a(X^k) is +-a[t] with t = j k^{-1} mod 2N (minus when t >= N);
    // k = 1 in multiply mode (every word is the owner's own)
    uint64_t v[ITEMS];
#pragma unroll
    for (int m = 0; m < ITEMS; ++m) {
      const uint32_t item = tau + m * T;
      const uint32_t c = item / Q, jl = item % Q, j = rank * Q + jl;
      const uint32_t t = (j * kinv) & (N - 1);
      v[m] = dsmem_ld_u64(dsmem_map(acc_s + (c * Q + (t % Q)) * 8u, t / Q));
    }
#pragma unroll
    for (int m = 0; m < ITEMS; ++m) {
      const uint32_t item = tau + m * T;
      const uint32_t c = item / Q, jl = item % Q, j = rank * Q + jl;
      const bool neg = ((j * kinv) & (TWO_N - 1)) >= N;
      const uint64_t w = neg ? 0ull - v[m] : v[m];
      if (!PTMUL && c == 1) {
        sig_b[jl] = w;
      } else {
        const uint32_t row0 = PTMUL ? c * dlev : 0;
        uint64_t cv = bits >= 64 ? w : (w + round_add) >> round_sh;
        for (int l = static_cast<int>(dlev) - 1; l >= 0; --l) {
          const uint64_t d = cv & Bmask;
          cv >>= a.base_log;
          int32_t ds = static_cast<int32_t>(d);
          if (d >= Bhalf) {
            ds -= static_cast<int32_t>(Bmask + 1);
            cv += 1;
          }
          dig[(row0 + l) * Q + jl] = ds;
        }
      }
    }
    cluster.sync();

    // ---- phase 2: digits x key_s for prime `rank` ----
    uint32_t oh[2][E];
    const uint32_t *kbase =
        a.keys + (static_cast<size_t>(s) * kPrimes + rank) * (static_cast<size_t>(a.level) * 2 * N);
    for (uint32_t r0 = 0; r0 < a.level; r0 += 2) {
      uint32_t x[2][E];
#pragma unroll
      for (int pp = 0; pp < 2; ++pp)
#pragma unroll
        for (int q = 0; q < E; ++q) {
          const uint32_t ad = dsmem_map(dig_s + ((r0 + pp) * Q + tau + (q % QE) * T) * 4u, q / QE);
          x[pp][q] = static_cast<uint32_t>(dsmem_ld_s32(ad) + static_cast<int32_t>(p));  // (0, 2p)
        }
      ntt_forward<LOGN, E, 2, 1>(x, tw, xb, tau, p);
      const uint4 *g = reinterpret_cast<const uint4 *>(kbase + static_cast<size_t>(r0) * 2 * N + E * tau);
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        uint32_t ga[E], gb[E];
#pragma unroll
        for (int kk = 0; kk < E / 4; ++kk) {
          const uint4 va = __ldg(g + (c * N) / 4 + kk), vb = __ldg(g + ((2 + c) * N) / 4 + kk);
          ga[4 * kk] = va.x; ga[4 * kk + 1] = va.y; ga[4 * kk + 2] = va.z; ga[4 * kk + 3] = va.w;
          gb[4 * kk] = vb.x; gb[4 * kk + 1] = vb.y; gb[4 * kk + 2] = vb.z; gb[4 * kk + 3] = vb.w;
        }
        if (c == 0) {
#pragma unroll
          for (int pp = 0; pp < 2; ++pp)
#pragma unroll
            for (int e = 0; e < E; ++e) x[pp][e] = cond_sub(x[pp][e], 8 * p);
        }
#pragma unroll
        for (int e = 0; e < E; ++e) {
          const uint64_t prod = static_cast<uint64_t>(x[0][e]) * ga[e] + static_cast<uint64_t>(x[1][e]) * gb[e];
          const uint32_t rr = redc(prod, p, p_inv);
          oh[c][e] = (r0 == 0) ? rr : cond_sub(oh[c][e] + rr, 4 * p);
        }
      }
    }
    ntt_inverse<LOGN, E, 2, 1>(oh, tw, xb, tau, p);
#pragma unroll
    for (int c = 0; c < 2; ++c)
#pragma unroll
      for (int q = 0; q < E; ++q) {
        const uint32_t y = oh[c][q];  // < 8p, CRT-scaled through the keys
        dsmem_st_u32(dsmem_map(res_s + ((rank * 2 + c) * Q + tau + (q % QE) * T) * 4u, q / QE), y);
      }
    cluster.sync();

    // ---- phase 3: c <- c + (0 - X_0, sigma_k(B) - X_1) on the owned quarter ----
#pragma unroll
    for (int m = 0; m < ITEMS; ++m) {
      const uint32_t item = tau + m * T;
      const uint32_t c = item / Q, jl = item % Q;
      uint64_t sum = 0;
      uint32_t ysum = 0;
#pragma unroll
      for (int pq = 0; pq < kPrimes; ++pq) {
        const uint32_t y = res[(pq * 2 + c) * Q + jl];
        sum += static_cast<uint64_t>(y) * a.cc.pr[pq].Mp_mod64;
        ysum += y >> 2;
      }
      const uint32_t u = crt_quotient(ysum);
      const uint64_t X = sum - static_cast<uint64_t>(u) * a.cc.M_mod64;
      if (PTMUL)
        acc[c * Q + jl] = X + ((c == 1 && a.plain_add) ? a.plain_add[rank * Q + jl] : 0ull);
      else
        acc[c * Q + jl] += (c == 1 ? sig_b[jl] : 0ull) - X;
    }
    cluster.sync();
  }

  uint64_t *gout = a.glwe_out + static_cast<size_t>(ct) * 2 * N;
#pragma unroll
  for (int m = 0; m < ITEMS; ++m) {
    const uint32_t item = tau + m * T;
    const uint32_t c = item / Q, jl = item % Q;
    gout[c * N + rank * Q + jl] = acc[c * Q + jl];
  }
  cluster.sync();
}

size_t trace_smem_bytes(uint32_t logN, uint32_t level) {
  const size_t N = size_t(1) << logN, Q = N / 4;
  size_t b = N * sizeof(uint2) + 3 * Q * sizeof(uint64_t) + kPrimes * 2 * Q * sizeof(uint32_t) +
             (N + N / 8) * sizeof(uint32_t) + level * Q * sizeof(int32_t);
  return (b + 15) & ~size_t(15);
}

template <int LOGN, bool PTMUL>
static cudaError_t launch_trace_t(const TraceArgs &a, cudaStream_t s) {
  auto kern = trace_kernel<LOGN, PTMUL>;
  const size_t smem = trace_smem_bytes(LOGN, a.level);
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(4 * a.batch, 1, 1);
  cfg.blockDim = dim3(TrShape<LOGN>::T, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 4;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, a);
}

template <bool PTMUL>
static cudaError_t launch_mode(const TraceArgs &a, uint32_t logN, cudaStream_t s) {
  switch (logN) {
    case 8: return launch_trace_t<8, PTMUL>(a, s);
    case 9: return launch_trace_t<9, PTMUL>(a, s);
    case 10: return launch_trace_t<10, PTMUL>(a, s);
    case 11: return launch_trace_t<11, PTMUL>(a, s);
    case 12: return launch_trace_t<12, PTMUL>(a, s);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_trace(const TraceArgs &a, uint32_t logN, cudaStream_t s) { return launch_mode<false>(a, logN, s); }

cudaError_t launch_plaintext_mul(const TraceArgs &a, uint32_t logN, cudaStream_t s) {
  return launch_mode<true>(a, logN, s);
}

// R <- (first ? 0 : R) + X^e r for `count` polynomials of N words (0 <= e < N):
// coefficient j of X^e r is r[j - e] for j >= e and -r[j - e + N] below.
__global__ void __launch_bounds__(256) monomial_acc_kernel(uint64_t *__restrict__ R, const uint64_t *__restrict__ r,
                                                          size_t words, uint32_t logN, uint32_t e, bool first) {
  const uint32_t N = 1u << logN;
  const size_t stride = static_cast<size_t>(gridDim.x) * blockDim.x;
  for (size_t i = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < words; i += stride) {
    const uint32_t j = static_cast<uint32_t>(i) & (N - 1);
    const size_t row = i - j;
    const uint64_t v = j >= e ? r[row + j - e] : 0ull - r[row + j - e + N];
    R[i] = first ? v : R[i] + v;
  }
}

cudaError_t launch_monomial_acc(uint64_t *R, const uint64_t *r, uint32_t count, uint32_t logN, uint32_t e, bool first,
                                cudaStream_t s) {
  const size_t words = static_cast<size_t>(count) << logN;
  if (words == 0) return cudaSuccess;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  size_t blocks = (words + 255) / 256;
  const size_t cap = static_cast<size_t>(sms > 0 ? sms : 1) * 8;
  if (blocks > cap) blocks = cap;
  monomial_acc_kernel<<<static_cast<unsigned>(blocks), 256, 0, s>>>(R, r, words, logN, e, first);
  return cudaGetLastError();
}

}  // namespace rosetta
