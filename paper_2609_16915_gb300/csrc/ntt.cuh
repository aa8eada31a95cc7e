// Negacyclic number-theoretic transforms of size N = 2^LOGN over one prime,
// distributed over N/E threads that each hold E = 8 or 16 residues in
// registers.
//
// Forward: Cooley-Tukey butterflies with the negacyclic twist merged into the
// twiddles (W[m] = psi^{bitrev(m)}, psi a primitive 2N-th root of unity);
// natural-order input, bit-reversed output.  Inverse: Gentleman-Sande
// butterflies, bit-reversed input, natural output, without the final N^{-1}
// (folded by the caller into its next constant).  The inverse twiddle of
// stage s, group g is psi^{-bitrev(2^s+g)} = -W[2^{s+1}-1-g], so one table
// serves both directions.
//
// The log2(N) stages are grouped into passes of log2(E) stages (the last pass
// takes what remains).  Within a pass each thread owns whole butterfly blocks
// and keeps them in registers; between passes the values are exchanged
// through a shared-memory buffer.  After the last forward pass thread t holds
// bit-reversed positions E t .. E t + E-1, which is exactly what the first
// inverse pass needs, so a pointwise product between the two transforms
// needs no exchange.
//
// Lazy ranges (primes below 2^28): forward input < 2p, output < 16p; inverse
// input < 4p, output < 8p.  See the butterflies for the per-stage invariants.
// With P31 (primes between 2^30 and 2^31, where 4p > 2^32 leaves no room for
// lazy growth) every input and output lies in [0, 2p).
#pragma once
#include <stdint.h>

#include "modarith.cuh"

namespace rosetta {

__host__ __device__ constexpr int ilog2(int x) { return x <= 1 ? 0 : 1 + ilog2(x >> 1); }

template <int LOGN, int E = 8>
struct NttShape {
  static_assert(E == 8 || E == 16, "8 or 16 values per thread");
  static constexpr int N = 1 << LOGN;
  static constexpr int T = N / E;                    // threads per transform
  static constexpr int RAD = ilog2(E);               // stages per full pass
  static constexpr int NPASS = (LOGN + RAD - 1) / RAD;
  static constexpr int LAST_H = LOGN - RAD * (NPASS - 1);
  static constexpr int XB_WORDS = N + N / 8;         // padded exchange buffer
  template <int PASS>
  __host__ __device__ static constexpr int h() { return PASS == NPASS - 1 ? LAST_H : RAD; }
};

// Exchange-buffer address: 4 pad words after every 32 keeps the scalar
// accesses of the passes (nearly) free of bank conflicts; the last pass, whose
// E consecutive words per thread stay 16-byte aligned, uses vector accesses.
__device__ __forceinline__ uint32_t xb_pad(uint32_t i) { return i + ((i >> 5) << 2); }
__host__ __device__ constexpr uint32_t xb_pad_c(uint32_t i) { return i + ((i >> 5) << 2); }

// Position (in the stage-ordered data array) of register slot e of thread
// tau during the pass that starts at stage S0 and spans H stages.  Blocks of
// 2^H elements have stride SIG = N >> (S0+H) and live in the stage-S0 group
// g of span N >> S0; a thread owns E >> H consecutive blocks.
template <int LOGN, int E, int S0, int H>
__device__ __forceinline__ uint32_t slot_index(uint32_t tau, int e) {
  constexpr uint32_t N = 1u << LOGN;
  constexpr uint32_t SIG = N >> (S0 + H);
  constexpr uint32_t SPAN = N >> S0;
  constexpr int NB = E >> H;
  const int b = e >> H;
  const int q = e & ((1 << H) - 1);
  const uint32_t beta = tau * NB + b;
  const uint32_t g = beta / SIG;
  const uint32_t i = beta % SIG;
  return g * SPAN + i + q * SIG;
}

// Forward (Cooley-Tukey) butterfly X' = X + wY, Y' = X - wY with t = wY in
// [0, 2p).  Without correction: inputs < a p give outputs < (a+2) p.  With
// correction X is first brought below 8p (valid for X < 16p), so the outputs
// are below 10p whatever Y was.
template <bool CORR>
__device__ __forceinline__ void ct_bfly(uint32_t &X, uint32_t &Y, uint2 w, uint32_t p, uint32_t two_p,
                                        uint32_t eight_p) {
  if (CORR) X = cond_sub(X, eight_p);
  const uint32_t t = shoup_mul(Y, w.x, w.y, p);
  Y = X - t + two_p;
  X = X + t;
}

// Butterflies for primes 2^30 < p < 2^31, every value in [0, 2p).  Forward:
// X' = x + t, Y' = x - t + p with x = X and t = wY both brought into [0, p)
// first (the Shoup product accepts any 32-bit Y, so Y needs no correction).
__device__ __forceinline__ void ct_bfly31(uint32_t &X, uint32_t &Y, uint2 w, uint32_t p) {
  const uint32_t x = cond_sub(X, p);
  const uint32_t t = cond_sub(shoup_mul(Y, w.x, w.y, p), p);
  X = x + t;
  Y = x - t + p;
}

// Inverse with twiddle -w: X' = x + y, Y' = (y - x + p) w, x and y the inputs
// brought into [0, p).
__device__ __forceinline__ void gs_bfly31(uint32_t &X, uint32_t &Y, uint2 w, uint32_t p) {
  const uint32_t x = cond_sub(X, p), y = cond_sub(Y, p);
  X = x + y;
  Y = shoup_mul(y - x + p, w.x, w.y, p);
}

// Stage s of the forward transform corrects X when s = 7, 11, 15, ...: the
// bounds run 2p -> 4p -> .. -> 16p after stage 6, then 10p (corrected),
// 12p, 14p, 16p, 10p (corrected), ...; 16p < 2^32.
__host__ __device__ constexpr bool fwd_stage_corrects(int s) { return s >= 7 && ((s - 7) % 4 == 0); }

// Inverse (Gentleman-Sande) butterfly with inverse twiddle -w:
// X' = X + Y, Y' = (X - Y)(-w) = (Y - X + 8p) w.  Inputs < 8p give
// X' < 16p, brought below 8p when corr, and Y' < 2p (16p < 2^32).
__device__ __forceinline__ void gs_bfly(uint32_t &X, uint32_t &Y, uint2 w, uint32_t p, uint32_t eight_p, bool corr) {
  const uint32_t s = X + Y;
  const uint32_t d = Y - X + eight_p;
  X = corr ? cond_sub(s, eight_p) : s;  // corr is a constant after unrolling
  Y = shoup_mul(d, w.x, w.y, p);
}

// Does inverse stage S (inside the pass (S0, H), U = S - S0) need the
// correction for the butterfly at register position q?  Both inputs of an
// inverse butterfly are outputs of the same kind (X' or Y') of stage S+1:
// X' outputs iff bit (H - U - 2) of q is 0.  Y' inputs (< 2p) give X' < 4p:
// no correction.  X' inputs are below 8p, or below 4p when their own
// butterfly at stage S+2 had Y' inputs (bit (H - U - 3) of q is 1, known
// when S+2 lies in the same pass): then X' < 8p needs no correction either.
// The first stage of a pass sees inputs of unknown kind and corrects, except
// the very first inverse stage (LAST pass), whose inputs are all below 4p.
template <bool LAST, int H, int U>
__host__ __device__ constexpr bool inv_corrects(int q) {
  if constexpr (U >= H - 1) {
    return !LAST;
  } else {
    if (((q >> (H - U - 2)) & 1) != 0) return false;
    if constexpr (U + 2 <= H - 1) {
      if (((q >> (H - U - 3)) & 1) == 1) return false;
    }
    return true;
  }
}

// Load CNT (a power of two) consecutive twiddle pairs starting at an index
// that is a multiple of CNT: one 8-byte or CNT/2 16-byte shared loads.
template <int CNT>
__device__ __forceinline__ void load_twiddles(const uint2 *__restrict__ tw, uint32_t start, uint2 (&w)[CNT]) {
  if constexpr (CNT == 1) {
    w[0] = tw[start];
  } else {
    const uint4 *p = reinterpret_cast<const uint4 *>(tw + start);
#pragma unroll
    for (int k = 0; k < CNT / 2; ++k) {
      const uint4 v = p[k];
      w[2 * k] = make_uint2(v.x, v.y);
      w[2 * k + 1] = make_uint2(v.z, v.w);
    }
  }
}

template <int LOGN, int E, int NP, int S0, int H, int U, bool P31>
__device__ __forceinline__ void fwd_stage(uint32_t (&x)[NP][E], const uint2 *__restrict__ tw, uint32_t tau,
                                          uint32_t p, uint32_t two_p, uint32_t eight_p) {
  constexpr uint32_t N = 1u << LOGN;
  constexpr uint32_t SIG = N >> (S0 + H);
  constexpr int NB = E >> H;
  constexpr int S = S0 + U;
  constexpr int HALF = 1 << (H - 1 - U);
  constexpr bool CORR = fwd_stage_corrects(S);
  if constexpr (SIG == 1) {
    // last pass: the thread's groups are consecutive, so are their twiddles
    constexpr int CNT = NB << U;
    uint2 w[CNT];
    load_twiddles<CNT>(tw, (1u << S) + tau * CNT, w);
#pragma unroll
    for (int b = 0; b < NB; ++b)
#pragma unroll
      for (int q = 0; q < (1 << H); ++q) {
        if (q & HALF) continue;
#pragma unroll
        for (int k = 0; k < NP; ++k) {
          if constexpr (P31)
            ct_bfly31(x[k][b * (1 << H) + q], x[k][b * (1 << H) + q + HALF], w[(b << U) + (q >> (H - U))], p);
          else
            ct_bfly<CORR>(x[k][b * (1 << H) + q], x[k][b * (1 << H) + q + HALF], w[(b << U) + (q >> (H - U))], p,
                          two_p, eight_p);
        }
      }
  } else {
#pragma unroll
    for (int b = 0; b < NB; ++b) {
      const uint32_t g = (tau * NB + b) / SIG;
#pragma unroll
      for (int q = 0; q < (1 << H); ++q) {
        if (q & HALF) continue;
        const uint2 w = tw[(1u << S) + (g << U) + (q >> (H - U))];
#pragma unroll
        for (int k = 0; k < NP; ++k) {
          if constexpr (P31)
            ct_bfly31(x[k][b * (1 << H) + q], x[k][b * (1 << H) + q + HALF], w, p);
          else
            ct_bfly<CORR>(x[k][b * (1 << H) + q], x[k][b * (1 << H) + q + HALF], w, p, two_p, eight_p);
        }
      }
    }
  }
}

template <int LOGN, int E, int NP, int S0, int H, int U, bool P31>
__device__ __forceinline__ void inv_stage(uint32_t (&x)[NP][E], const uint2 *__restrict__ tw, uint32_t tau,
                                          uint32_t p, uint32_t eight_p) {
  constexpr bool LAST = (S0 + H == LOGN);  // the pass the inverse starts with
  constexpr uint32_t N = 1u << LOGN;
  constexpr uint32_t SIG = N >> (S0 + H);
  constexpr int NB = E >> H;
  constexpr int S = S0 + U;
  constexpr int HALF = 1 << (H - 1 - U);
  if constexpr (SIG == 1) {
    // last pass: groups G in [tau*CNT, (tau+1)*CNT) use the descending run
    // W[2^{s+1}-1-G], which starts at 2^{s+1} - (tau+1)*CNT
    constexpr int CNT = NB << U;
    uint2 w[CNT];
    load_twiddles<CNT>(tw, (2u << S) - (tau + 1) * CNT, w);
#pragma unroll
    for (int b = 0; b < NB; ++b)
#pragma unroll
      for (int q = 0; q < (1 << H); ++q) {
        if (q & HALF) continue;
        const int idx = CNT - 1 - ((b << U) + (q >> (H - U)));
#pragma unroll
        for (int k = 0; k < NP; ++k) {
          if constexpr (P31)
            gs_bfly31(x[k][b * (1 << H) + q], x[k][b * (1 << H) + q + HALF], w[idx], p);
          else
            gs_bfly(x[k][b * (1 << H) + q], x[k][b * (1 << H) + q + HALF], w[idx], p, eight_p,
                    inv_corrects<LAST, H, U>(q));
        }
      }
  } else {
#pragma unroll
    for (int b = 0; b < NB; ++b) {
      const uint32_t g = (tau * NB + b) / SIG;
#pragma unroll
      for (int q = 0; q < (1 << H); ++q) {
        if (q & HALF) continue;
        const uint32_t G = (g << U) + (q >> (H - U));
        const uint2 w = tw[(2u << S) - 1u - G];
#pragma unroll
        for (int k = 0; k < NP; ++k) {
          if constexpr (P31)
            gs_bfly31(x[k][b * (1 << H) + q], x[k][b * (1 << H) + q + HALF], w, p);
          else
            gs_bfly(x[k][b * (1 << H) + q], x[k][b * (1 << H) + q + HALF], w, p, eight_p,
                    inv_corrects<LAST, H, U>(q));
        }
      }
    }
  }
}

template <int LOGN, int E, int NP, int S0, int H, bool P31, int U = 0>
__device__ __forceinline__ void fwd_pass(uint32_t (&x)[NP][E], const uint2 *tw, uint32_t tau, uint32_t p,
                                         uint32_t two_p, uint32_t eight_p) {
  fwd_stage<LOGN, E, NP, S0, H, U, P31>(x, tw, tau, p, two_p, eight_p);
  if constexpr (U + 1 < H) fwd_pass<LOGN, E, NP, S0, H, P31, U + 1>(x, tw, tau, p, two_p, eight_p);
}

template <int LOGN, int E, int NP, int S0, int H, bool P31, int U = H - 1>
__device__ __forceinline__ void inv_pass(uint32_t (&x)[NP][E], const uint2 *tw, uint32_t tau, uint32_t p,
                                         uint32_t eight_p) {
  inv_stage<LOGN, E, NP, S0, H, U, P31>(x, tw, tau, p, eight_p);
  if constexpr (U > 0) inv_pass<LOGN, E, NP, S0, H, P31, U - 1>(x, tw, tau, p, eight_p);
}

// A pass whose butterfly groups span S elements keeps the data of every run of
// G = max(1, S / (32 E)) consecutive warps inside one aligned range of 32 E G
// elements, so an exchange out of (or into) that pass only has to
// synchronise those G warps: the warp itself when S <= 32 E, a named barrier
// over 32 G threads in between, the whole CTA when G covers it.
template <int LOGN, int E, int S0>
__host__ __device__ constexpr int pass_group_warps() {
  return (1 << (LOGN - S0)) <= 32 * E ? 1 : (1 << (LOGN - S0)) / (32 * E);
}

template <int G, int WARPS>
__device__ __forceinline__ void group_sync(uint32_t tau) {
  if constexpr (G <= 1) {
    __syncwarp();
  } else if constexpr (G >= WARPS) {
    __syncthreads();
  } else {
    static_assert(WARPS / G <= 15, "named barriers 1..15");
    asm volatile("bar.sync %0, %1;" ::"r"(1u + (tau >> 5) / G), "r"(32 * G) : "memory");
  }
}

// Padded address of slot e of thread tau in the pass (S0, H), split as a
// per-thread base plus a compile-time offset: for every pass shape the low
// five bits of base and offset never carry, so pad(base + off) =
// pad(base) + pad(off).  Non-last passes have one block per thread
// (base = g*SPAN + i, offset e*SIG); in the last pass a thread's slots are
// the E consecutive positions E*tau + e.
template <int LOGN, int E, int S0, int H>
__device__ __forceinline__ uint32_t xb_base(uint32_t tau) {
  constexpr uint32_t N = 1u << LOGN, SIG = N >> (S0 + H), SPAN = N >> S0;
  if constexpr (SIG == 1) {
    return xb_pad(E * tau);
  } else {
    static_assert((1 << H) == E, "only the last pass is shorter than a full pass");
    return xb_pad((tau / SIG) * SPAN + tau % SIG);
  }
}

template <int LOGN, int E, int S0, int H>
__host__ __device__ constexpr uint32_t xb_off(int e) {
  constexpr uint32_t N = 1u << LOGN, SIG = N >> (S0 + H);
  return xb_pad_c(SIG == 1 ? static_cast<uint32_t>(e) : static_cast<uint32_t>(e) * SIG);
}

// Store / load one thread's E slots of the pass (S0, H).  In the last pass the
// E consecutive words are 16-byte aligned: E/4 vector accesses.
template <int LOGN, int E, int S0, int H>
__device__ __forceinline__ void xb_store(uint32_t *buf, const uint32_t (&v)[E], uint32_t tau) {
  uint32_t *b = buf + xb_base<LOGN, E, S0, H>(tau);
  if constexpr (S0 + H == LOGN) {
    uint4 *p = reinterpret_cast<uint4 *>(b);
#pragma unroll
    for (int k = 0; k < E / 4; ++k) p[k] = make_uint4(v[4 * k], v[4 * k + 1], v[4 * k + 2], v[4 * k + 3]);
  } else {
#pragma unroll
    for (int e = 0; e < E; ++e) b[xb_off<LOGN, E, S0, H>(e)] = v[e];
  }
}

template <int LOGN, int E, int S0, int H>
__device__ __forceinline__ void xb_load(const uint32_t *buf, uint32_t (&v)[E], uint32_t tau) {
  const uint32_t *b = buf + xb_base<LOGN, E, S0, H>(tau);
  if constexpr (S0 + H == LOGN) {
    const uint4 *p = reinterpret_cast<const uint4 *>(b);
#pragma unroll
    for (int k = 0; k < E / 4; ++k) {
      const uint4 a = p[k];
      v[4 * k] = a.x;
      v[4 * k + 1] = a.y;
      v[4 * k + 2] = a.z;
      v[4 * k + 3] = a.w;
    }
  } else {
#pragma unroll
    for (int e = 0; e < E; ++e) v[e] = b[xb_off<LOGN, E, S0, H>(e)];
  }
}

// Move NP register sets from the layout of pass A to that of pass B through
// the exchange buffer xb (XBUF polynomials of NttShape::XB_WORDS words each).
// The leading barrier protects xb from readers of the previous exchange; both
// barriers cover only the warps whose data the exchange mixes.
template <int LOGN, int E, int NP, int XBUF, int S0A, int HA, int S0B, int HB>
__device__ __forceinline__ void exchange(uint32_t (&x)[NP][E], uint32_t *xb, uint32_t tau) {
  constexpr int W = NttShape<LOGN, E>::XB_WORDS;
  constexpr int G = pass_group_warps<LOGN, E, (S0A < S0B ? S0A : S0B)>();
  constexpr int WARPS = NttShape<LOGN, E>::T / 32 > 0 ? NttShape<LOGN, E>::T / 32 : 1;
  static_assert(XBUF == 1 || XBUF == NP, "exchange buffer must hold one or all polynomials");
  if constexpr (XBUF == NP) {
    group_sync<G, WARPS>(tau);
#pragma unroll
    for (int k = 0; k < NP; ++k) xb_store<LOGN, E, S0A, HA>(xb + k * W, x[k], tau);
    group_sync<G, WARPS>(tau);
#pragma unroll
    for (int k = 0; k < NP; ++k) xb_load<LOGN, E, S0B, HB>(xb + k * W, x[k], tau);
  } else {
#pragma unroll
    for (int k = 0; k < NP; ++k) {
      group_sync<G, WARPS>(tau);
      xb_store<LOGN, E, S0A, HA>(xb, x[k], tau);
      group_sync<G, WARPS>(tau);
      xb_load<LOGN, E, S0B, HB>(xb, x[k], tau);
    }
  }
}

// Forward transform of NP polynomials held as x[k][e] = element
// slot_index<LOGN,E,0,RAD>(tau, e) = tau + e*N/E of polynomial k.
template <int LOGN, int E, int NP, int XBUF, bool P31 = false, int PASS = 0>
__device__ __forceinline__ void ntt_forward(uint32_t (&x)[NP][E], const uint2 *tw, uint32_t *xb, uint32_t tau,
                                            uint32_t p) {
  using S = NttShape<LOGN, E>;
  constexpr int S0 = S::RAD * PASS;
  constexpr int H = S::template h<PASS>();
  fwd_pass<LOGN, E, NP, S0, H, P31>(x, tw, tau, p, 2 * p, 8 * p);
  if constexpr (PASS + 1 < S::NPASS) {
    exchange<LOGN, E, NP, XBUF, S0, H, S0 + S::RAD, S::template h<PASS + 1>()>(x, xb, tau);
    ntt_forward<LOGN, E, NP, XBUF, P31, PASS + 1>(x, tw, xb, tau, p);
  }
}

// Inverse transform (without the N^{-1} factor).  Input: x[k][e] holds
// bit-reversed position E*tau + e; output: natural position tau + e*N/E.
template <int LOGN, int E, int NP, int XBUF, bool P31 = false, int PASS = NttShape<LOGN, E>::NPASS - 1>
__device__ __forceinline__ void ntt_inverse(uint32_t (&x)[NP][E], const uint2 *tw, uint32_t *xb, uint32_t tau,
                                            uint32_t p) {
  using S = NttShape<LOGN, E>;
  constexpr int S0 = S::RAD * PASS;
  constexpr int H = S::template h<PASS>();
  inv_pass<LOGN, E, NP, S0, H, P31>(x, tw, tau, p, 8 * p);
  if constexpr (PASS > 0) {
    exchange<LOGN, E, NP, XBUF, S0, H, S0 - S::RAD, S::RAD>(x, xb, tau);
    ntt_inverse<LOGN, E, NP, XBUF, P31, PASS - 1>(x, tw, xb, tau, p);
  }
}

}  // namespace rosetta
