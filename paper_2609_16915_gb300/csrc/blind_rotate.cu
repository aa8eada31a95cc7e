// Blind rotation (modulus switch -> n CMux steps -> sample extraction) for a
// batch of LWE ciphertexts, one thread-block cluster of four CTAs per
// ciphertext.
//
// Construction (Background, "TFHE Scheme", PBS): the LUT is written into a
// test polynomial v, the accumulator starts as the trivial GLWE
// (0, X^{-b~} v) and every CMux step i multiplies it by X^{a~_i s_i} through
// the external product with the GGSW BSK_i:
//     ACC <- ACC + BSK_i (x) (X^{a~_i} ACC - ACC).
// The external product decomposes each coefficient of the rotated difference
// into signed digits and forms sum_r D_r * BSK_i[r][c] in Z_{2^64}[X]/(X^N+1).
// Those products are computed exactly: the integer value of every output
// coefficient is below M/2 with M the product of four 28-bit NTT primes, so
// four negacyclic NTTs, a pointwise multiply-accumulate per prime and an
// explicit CRT (X = sum_q y_q M/p_q - round(sum_q y_q/p_q) M, evaluated mod
// 2^64) give the same words as the schoolbook product.
//
// Work split.  CTA r of the cluster (r = 0..3) does all transforms for prime
// r and owns coefficients [rN/4, (r+1)N/4) of both accumulator polynomials.
// One CMux step is three phases separated by cluster barriers:
//   1. each owner forms the rotated difference for its quarter (reading the
//      rotated source coefficient from whichever CTA owns it, through
//      distributed shared memory) and writes its gadget digits locally, in
//      packed groups of four per thread;
//   2. each prime-CTA gathers all digits (one vector DSMEM load per owner
//      and thread), runs forward NTTs two polynomials at a time, multiplies
//      by the transform-domain BSK_i (streamed from global memory with
//      16-byte loads, Montgomery form), runs the two inverse NTTs and leaves
//      the CRT-scaled residues of each owner's quarter in its own exchange
//      buffer (one vector store per owner and thread);
//   3. each owner reads the four residues of its coefficients from the four
//      prime-CTAs (one vector DSMEM load each), combines them (explicit CRT)
//      and adds the result to the accumulator.
// Every cross-CTA read follows a write to the writer's own shared memory, so
// the step's barriers order shared memory only (cluster_sync_shared).
#include <cooperative_groups.h>

#include <type_traits>

#include "check.cuh"
#include "dsmem.cuh"
#include "internal.h"
#include "ntt.cuh"

namespace rosetta {
namespace cg = cooperative_groups;

// One exchange buffer per polynomial of a pair only where shared memory is
// plentiful; larger rings share one buffer to keep more CTAs resident.
__host__ __device__ constexpr int br_xbuf(int logN) { return logN <= 10 ? 2 : 1; }

// Exchange-buffer words: the transforms' XBUF x (N + N/8), and at least 2N
// (16 T) for the outgoing residues, four groups of four words per thread.
__host__ __device__ constexpr int br_xb_words(int logN) {
  return br_xbuf(logN) * ((1 << logN) + (1 << logN) / 8) > 2 * (1 << logN)
             ? br_xbuf(logN) * ((1 << logN) + (1 << logN) / 8)
             : 2 * (1 << logN);
}

// Values per thread in the transforms.  16 halves the CTA-wide exchanges but
// also the warps per SM; measured on GB300 it is slower at every ring size
// (N = 2048: 309 vs 276 ms, 4096: 822 vs 782 ms, 8192: 14.0 vs 12.8 s for the
// full batches), so 8 is used throughout.
__host__ __device__ constexpr int br_e(int) { return 8; }

template <int LOGN>
struct BrShape {
  static constexpr int N = 1 << LOGN;
  static constexpr int E = br_e(LOGN);
  static constexpr int T = N / E;                      // threads per CTA
  static constexpr int Q = N / 4;                      // coefficients owned per CTA
  static constexpr int ITEMS = 2 * Q / T;              // owned (component, coefficient) pairs per thread
  static constexpr int QE = E / 4;                     // first-pass slots per owner quarter
  static constexpr int XBUF = br_xbuf(LOGN);            // exchange buffers (polys)
  // resident CTAs per SM the register allocation must allow (shared memory
  // allows the same: 4 x 46 KB at N = 2048, 2 x 90 KB at 4096)
  static constexpr int MIN_CTAS = (LOGN <= 11) ? 4 : (LOGN == 12 ? 2 : 1);
};

// LEV > 0 fixes the gadget level count at compile time (the common sets:
// straight-line digit and key loops); LEV = 0 reads it from the arguments.
template <int LOGN, bool DIG16, int LEV>
__global__ void __launch_bounds__(BrShape<LOGN>::T, BrShape<LOGN>::MIN_CTAS) blind_rotate_kernel(const BrArgs a) {
  using B = BrShape<LOGN>;
  using S = NttShape<LOGN, B::E>;
  using DigT = typename std::conditional<DIG16, int16_t, int32_t>::type;
  constexpr uint32_t N = B::N, T = B::T, Q = B::Q;
  constexpr int E = B::E, ITEMS = B::ITEMS, QE = B::QE;
  constexpr uint32_t TWO_N = 2 * N;

  cg::cluster_group cluster = cg::this_cluster();
  const uint32_t rank = cluster.block_rank();
  const uint32_t ct = blockIdx.x / 4;
  const uint32_t tau = threadIdx.x;
  if (!dbg_ok(ct < a.batch, a.err_flag)) return;  // the whole cluster shares ct

  extern __shared__ __align__(16) unsigned char smem[];
  uint2 *tw = reinterpret_cast<uint2 *>(smem);                   // [N]
  uint64_t *acc = reinterpret_cast<uint64_t *>(tw + N);          // [2][Q]
  // [XBUF][XB_WORDS] for the transforms; after the inverse transforms the
  // outgoing residues [owner][T][2 comp][QE halves]
  uint32_t *xb = reinterpret_cast<uint32_t *>(acc + 2 * Q);
  static_assert(br_xb_words(LOGN) >= B::XBUF * S::XB_WORDS, "exchange buffer");
  DigT *dig = reinterpret_cast<DigT *>(xb + br_xb_words(LOGN));  // [l row pairs][T][2][QE]
  const uint32_t level = LEV > 0 ? static_cast<uint32_t>(LEV) : a.level;
  uint16_t *atil = reinterpret_cast<uint16_t *>(dig + 2 * level * Q);  // [n+1]

  const uint32_t p = a.cc.pr[rank].p;
  const uint32_t p_inv = a.cc.pr[rank].p_inv;

  // ---- set-up: twiddles, modulus switch, accumulator ----
  for (uint32_t m = tau; m < N; m += T) tw[m] = a.tw[rank * N + m];
  const uint64_t *lwe = a.lwe_in + static_cast<size_t>(ct) * (a.n + 1);
  constexpr uint32_t SH = 63 - LOGN;  // 64 - log2(2N)
  for (uint32_t i = tau; i <= a.n; i += T)
    atil[i] = static_cast<uint16_t>(((lwe[i] + (1ull << (SH - 1))) >> SH) & (TWO_N - 1));
  __syncthreads();
  {
    const uint32_t btil = atil[a.n];
    if (a.glwe_in) {
      // encrypted test polynomial: ACC = X^{-b~} (A, B) for this ciphertext
      const uint64_t *gin = a.glwe_in + static_cast<size_t>(ct) * 2 * N;
#pragma unroll
      for (int m = 0; m < ITEMS; ++m) {
        const uint32_t item = tau + m * T;
        const uint32_t c = item / Q, jl = item % Q, j = rank * Q + jl;
        const uint32_t e = (j + btil) & (TWO_N - 1);
        const uint64_t v = gin[c * N + (e & (N - 1))];
        acc[c * Q + jl] = (e >= N) ? 0ull - v : v;
      }
    } else {
      // trivial GLWE (0, X^{-b~} v) of the test polynomial of this ciphertext's LUT
      uint32_t li = 0;
      if (a.lut_index) {
        li = a.lut_index[ct];
        if (li >= a.num_luts) {  // never read outside the LUT array
          if (tau == 0 && rank == 0 && a.err_flag) atomicExch(a.err_flag, 1u);
          li = 0;
        }
      }
      const uint64_t *lut = a.lut + (static_cast<size_t>(li) << a.msg_bits);
      const uint32_t box = N >> a.msg_bits, h = box >> 1;
#pragma unroll
      for (int m = 0; m < ITEMS; ++m) {
        const uint32_t item = tau + m * T;
        const uint32_t c = item / Q, jl = item % Q, j = rank * Q + jl;
        if (c == 0) {
          acc[jl] = 0;
        } else {
          // (X^{2N - b~} v)[j] = +-v[t], t = (j + b~) mod 2N folded into [0, N)
          const uint32_t e = (j + btil) & (TWO_N - 1);
          const uint32_t t = e & (N - 1);
          const uint64_t v = (t < N - h) ? lut[(t + h) / box] : (0ull - lut[0]);
          acc[Q + jl] = (e >= N) ? 0ull - v : v;
        }
      }
    }
  }
  cluster.sync();

  // 32-bit shared-memory addresses; mapa turns them into the same location
  // in another CTA of the cluster
  const uint32_t acc_s = smem_addr(acc), dig_s = smem_addr(dig), xb_s = smem_addr(xb);
  const uint32_t L2 = 2 * level;
  const uint32_t bits = a.base_log * level;
  const uint64_t Bmask = (1ull << a.base_log) - 1;
  const uint64_t Bhalf = 1ull << (a.base_log - 1);
  const uint64_t round_add = bits >= 64 ? 0 : (1ull << (63 - bits));
  const uint32_t round_sh = bits >= 64 ? 0 : 64 - bits;

  // Packed exchange layouts.  Owner thread tau holds the items (c, jl) =
  // (m / QE, tau + (m % QE) T), m < ITEMS = 2 QE, and prime thread tau needs
  // from owner o exactly the coefficients tau + h T (h < QE) of both
  // components: so digits are stored as [row pair][tau][row parity][h] in
  // their owner and residues as [owner][tau][component][h] in their
  // prime-CTA, and every transfer between a pair of threads is one 2 QE-word
  // vector access.
  static_assert(ITEMS == 2 * QE, "one packed group of 2 QE items per thread");
  constexpr uint32_t GRP = 2 * QE;  // words per packed group
  const uint32_t dig_t = dig_s + tau * GRP * static_cast<uint32_t>(sizeof(DigT));
  const uint32_t res_t = xb_s + (rank * T + tau) * GRP * 4u;  // this owner's group in every prime-CTA
  // With one gadget level and N <= 2048 the remote bases of this thread's
  // digit and residue groups in each CTA are kept across the steps (measured
  // 1.5 % faster at N = 2048); elsewhere the registers are needed for the
  // transforms.
  constexpr bool HOIST = (LEV == 1 && LOGN <= 11);
  uint32_t dig_r[4], res_r[4];
  if constexpr (HOIST) {
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      dig_r[r] = dsmem_map(dig_t, r);
      res_r[r] = dsmem_map(res_t, r);
    }
  }
  for (uint32_t i = 0; i < a.n; ++i) {
    const uint32_t at = atil[i];
    if (at == 0) continue;  // X^0 ACC - ACC = 0: the step adds nothing

    // ---- phase 1: rotated difference and gadget digits of the owned quarter ----
    // (X^a P)[j] = +-P[(j - a) mod 2N]; all remote words are requested
    // before any is used so their latencies overlap
    uint64_t v[ITEMS];
#pragma unroll
    for (int m = 0; m < ITEMS; ++m) {
      const uint32_t item = tau + m * T;
      const uint32_t c = item / Q, jl = item % Q, j = rank * Q + jl;
      const uint32_t e = (j + TWO_N - at) & (N - 1);
      v[m] = dsmem_ld_u64(dsmem_map(acc_s + (c * Q + (e % Q)) * 8u, e / Q));
    }
    // with a compile-time level the packed groups are assembled in registers
    // and written with one vector store each
    constexpr int NGRP = LEV > 0 ? LEV : 1;
    int32_t grp[NGRP][GRP];
#pragma unroll
    for (int m = 0; m < ITEMS; ++m) {
      const uint32_t item = tau + m * T;
      const uint32_t c = item / Q, jl = item % Q, j = rank * Q + jl;
      const bool neg = ((j + TWO_N - at) & (TWO_N - 1)) >= N;
      const uint64_t diff = (neg ? 0ull - v[m] : v[m]) - acc[c * Q + jl];
      uint64_t cv = bits >= 64 ? diff : (diff + round_add) >> round_sh;
#pragma unroll
      for (int l = static_cast<int>(level) - 1; l >= 0; --l) {
        const uint64_t d = cv & Bmask;
        cv >>= a.base_log;
        int32_t ds = static_cast<int32_t>(d);
        if (d >= Bhalf) {
          ds -= static_cast<int32_t>(Bmask + 1);
          cv += 1;
        }
        const uint32_t r = c * level + l;  // row; h = m % QE
        if constexpr (LEV > 0)
          grp[r >> 1][(r & 1) * QE + (m % QE)] = ds;
        else
          dig[(((r >> 1) * T + tau) * 2 + (r & 1)) * QE + (m % QE)] = static_cast<DigT>(ds);
      }
    }
    if constexpr (LEV > 0) {
      static_assert(GRP == 4, "four digits per group");
#pragma unroll
      for (int P = 0; P < NGRP; ++P) {
        DigT *g = dig + (P * T + tau) * GRP;
        if constexpr (DIG16)
          *reinterpret_cast<uint2 *>(g) =
              make_uint2((static_cast<uint32_t>(grp[P][0]) & 0xFFFFu) | (static_cast<uint32_t>(grp[P][1]) << 16),
                         (static_cast<uint32_t>(grp[P][2]) & 0xFFFFu) | (static_cast<uint32_t>(grp[P][3]) << 16));
        else
          *reinterpret_cast<uint4 *>(g) = make_uint4(static_cast<uint32_t>(grp[P][0]), static_cast<uint32_t>(grp[P][1]),
                                                     static_cast<uint32_t>(grp[P][2]), static_cast<uint32_t>(grp[P][3]));
      }
    }
    cluster_sync_shared();

    // ---- phase 2: transforms and pointwise products for prime `rank` ----
    uint32_t oh[2][E];
    const size_t kblk = static_cast<size_t>(L2) * 2 * N;  // words of one step's key block per prime
    const uint32_t *gbase = a.bsk + (static_cast<size_t>(i) * kPrimes + rank) * kblk;
    const bool key_ok = dbg_ok(a.bsk_words == 0 || (static_cast<size_t>(i) * kPrimes + rank + 1) * kblk <= a.bsk_words,
                               a.err_flag);
    // The row pairs stay a rolled loop: unrolled, two levels at N = 4096
    // spill 56 bytes per thread (pulled residues hold more registers across
    // phase 2) and three levels at N = 8192 were 10 % slower.
#pragma unroll 1
    for (uint32_t r0 = 0; r0 < L2; r0 += 2) {
      // first-pass slot q of thread tau is coefficient tau + q N/E, owned by
      // CTA o = q / QE at local index tau + (q % QE) T: one packed group of
      // the row pair per owner
      uint32_t x[2][E];
      const uint32_t pair_off = (r0 >> 1) * T * GRP * static_cast<uint32_t>(sizeof(DigT));
#pragma unroll
      for (int o = 0; o < 4; ++o) {
        const uint32_t ad = (HOIST ? dig_r[o] : dsmem_map(dig_t, o)) + pair_off;
        int32_t d[GRP];
        if constexpr (DIG16) {
          static_assert(GRP == 4, "four 16-bit digits per group");
          const uint2 w = dsmem_ld_v2_u32(ad);
          d[0] = static_cast<int16_t>(w.x & 0xFFFFu);
          d[1] = static_cast<int16_t>(w.x >> 16);
          d[2] = static_cast<int16_t>(w.y & 0xFFFFu);
          d[3] = static_cast<int16_t>(w.y >> 16);
        } else {
          static_assert(GRP == 4, "four 32-bit digits per group");
          const uint4 w = dsmem_ld_v4_u32(ad);
          d[0] = static_cast<int32_t>(w.x);
          d[1] = static_cast<int32_t>(w.y);
          d[2] = static_cast<int32_t>(w.z);
          d[3] = static_cast<int32_t>(w.w);
        }
#pragma unroll
        for (int pp = 0; pp < 2; ++pp)
#pragma unroll
          for (int h = 0; h < QE; ++h)
            x[pp][o * QE + h] = static_cast<uint32_t>(d[pp * QE + h] + static_cast<int32_t>(p));  // in (0, 2p)
      }
      ntt_forward<LOGN, E, 2, B::XBUF>(x, tw, xb, tau, p);
      // BSK_i words of this prime for rows r0, r0+1, E per thread and
      // component, contiguous across the CTA (16-byte loads)
      const uint4 *g = reinterpret_cast<const uint4 *>(gbase + static_cast<size_t>(r0) * 2 * N + E * tau);
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        uint32_t ga[E], gb[E];
#pragma unroll
        for (int k = 0; k < E / 4; ++k) {
          const uint4 va = key_ok ? __ldg(g + (c * N) / 4 + k) : make_uint4(0u, 0u, 0u, 0u);
          const uint4 vb = key_ok ? __ldg(g + ((2 + c) * N) / 4 + k) : make_uint4(0u, 0u, 0u, 0u);
          ga[4 * k] = va.x; ga[4 * k + 1] = va.y; ga[4 * k + 2] = va.z; ga[4 * k + 3] = va.w;
          gb[4 * k] = vb.x; gb[4 * k + 1] = vb.y; gb[4 * k + 2] = vb.z; gb[4 * k + 3] = vb.w;
        }
        if (c == 0) {
#pragma unroll
          for (int pp = 0; pp < 2; ++pp)
#pragma unroll
            for (int e = 0; e < E; ++e) x[pp][e] = cond_sub(x[pp][e], 8 * p);  // < 16p -> < 8p
        }
#pragma unroll
        for (int e = 0; e < E; ++e) {
          // forward outputs < 8p, BSK words < p in Montgomery form: the pair
          // sum stays below 16 p^2 < p * 2^32
          const uint64_t prod = static_cast<uint64_t>(x[0][e]) * ga[e] + static_cast<uint64_t>(x[1][e]) * gb[e];
          const uint32_t rr = redc(prod, p, p_inv);  // (0, 2p)
          oh[c][e] = (r0 == 0) ? rr : cond_sub(oh[c][e] + rr, 4 * p);
        }
      }
    }
    ntt_inverse<LOGN, E, 2, B::XBUF>(oh, tw, xb, tau, p);
    __syncthreads();  // every exchange read done: the buffer takes the outgoing residues
    // CRT-scaled residues (< 8p; the keys carry the CRT factor), one packed
    // group (component, h) per owner
#pragma unroll
    for (int o = 0; o < 4; ++o) {
      static_assert(GRP == 4, "four residues per group");
      uint32_t y[4];
#pragma unroll
      for (int c = 0; c < 2; ++c)
#pragma unroll
        for (int h = 0; h < QE; ++h) y[c * QE + h] = oh[c][o * QE + h];
      *reinterpret_cast<uint4 *>(xb + (o * T + tau) * GRP) = make_uint4(y[0], y[1], y[2], y[3]);
    }
    cluster_sync_shared();

    // ---- phase 3: explicit CRT of the owned quarter, accumulate ----
    // item m of this thread is entry m of its packed group in every prime-CTA
    uint32_t yq[kPrimes][GRP];
#pragma unroll
    for (int pq = 0; pq < kPrimes; ++pq) {
      const uint4 w = dsmem_ld_v4_u32(HOIST ? res_r[pq] : dsmem_map(res_t, pq));
      yq[pq][0] = w.x;
      yq[pq][1] = w.y;
      yq[pq][2] = w.z;
      yq[pq][3] = w.w;
    }
#pragma unroll
    for (int m = 0; m < ITEMS; ++m) {
      const uint32_t item = tau + m * T;
      const uint32_t c = item / Q, jl = item % Q;
      uint64_t s = 0;
      uint32_t ysum = 0;
#pragma unroll
      for (int pq = 0; pq < kPrimes; ++pq) {
        const uint32_t y = yq[pq][m];
        s += static_cast<uint64_t>(y) * a.cc.pr[pq].Mp_mod64;
        ysum += y >> 2;  // y < 8p < 2^31: the sum stays below 2^31
      }
      const uint32_t u = crt_quotient(ysum);
      acc[c * Q + jl] += s - static_cast<uint64_t>(u) * a.cc.M_mod64;
    }
    cluster_sync_shared();
  }

  if (a.glwe_out) {
    // ---- the rotated accumulator itself ----
    uint64_t *gout = a.glwe_out + static_cast<size_t>(ct) * 2 * N;
#pragma unroll
    for (int m = 0; m < ITEMS; ++m) {
      const uint32_t item = tau + m * T;
      const uint32_t c = item / Q, jl = item % Q;
      gout[c * N + rank * Q + jl] = acc[c * Q + jl];
    }
  } else {
    // ---- sample extraction of the constant coefficient ----
    uint64_t *out = a.lwe_big_out + static_cast<size_t>(ct) * (N + 1);
#pragma unroll
    for (int m = 0; m < ITEMS; ++m) {
      const uint32_t item = tau + m * T;
      const uint32_t c = item / Q, jl = item % Q, j = rank * Q + jl;
      if (c == 0) {
        out[j == 0 ? 0 : N - j] = (j == 0) ? acc[jl] : 0ull - acc[jl];
      } else if (j == 0) {
        out[N] = acc[Q];
      }
    }
  }
  cluster.sync();
}

size_t br_smem_bytes(uint32_t logN, uint32_t level, uint32_t n, bool dig16) {
  const size_t N = size_t(1) << logN, Q = N / 4;
  size_t b = N * sizeof(uint2) + 2 * Q * sizeof(uint64_t) + br_xb_words(static_cast<int>(logN)) * sizeof(uint32_t) +
             2 * level * Q * (dig16 ? 2 : 4) + (n + 1) * sizeof(uint16_t);
  return (b + 15) & ~size_t(15);
}

template <int LOGN, bool DIG16, int LEV>
static cudaError_t launch_br_t(const BrArgs &a, cudaStream_t s) {
  auto kern = blind_rotate_kernel<LOGN, DIG16, LEV>;
  const size_t smem = br_smem_bytes(LOGN, a.level, a.n, DIG16);
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(4 * a.batch, 1, 1);
  cfg.blockDim = dim3(BrShape<LOGN>::T, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 4;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeClusterSchedulingPolicyPreference;
  attr[1].val.clusterSchedulingPolicyPreference = br_cluster_policy(kern, BrShape<LOGN>::T, smem, cfg.gridDim.x);
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, a);
}

template <int LOGN, bool DIG16>
static cudaError_t launch_br_lev(const BrArgs &a, cudaStream_t s) {
  if constexpr (LOGN >= 11) {
    // (a compile-time level also lets phase 1 write its packed digit groups
    // with one vector store each)
    switch (a.level) {
      case 1: return launch_br_t<LOGN, DIG16, 1>(a, s);
      case 2: return launch_br_t<LOGN, DIG16, 2>(a, s);
      case 3: return launch_br_t<LOGN, DIG16, 3>(a, s);
      default: break;
    }
  }
  return launch_br_t<LOGN, DIG16, 0>(a, s);
}

cudaError_t launch_blind_rotate(const BrArgs &a, uint32_t logN, bool dig16, cudaStream_t s) {
  if (a.primes == kPrimes31) return launch_blind_rotate3(a, logN, s);
  if (a.primes != kPrimes) return cudaErrorInvalidValue;
#define ROSETTA_BR_CASE(L)                                                        \
  case L:                                                                         \
    return dig16 ? launch_br_lev<L, true>(a, s) : launch_br_lev<L, false>(a, s);
  switch (logN) {
    ROSETTA_BR_CASE(8)
    ROSETTA_BR_CASE(9)
    ROSETTA_BR_CASE(10)
    ROSETTA_BR_CASE(11)
    ROSETTA_BR_CASE(12)
    ROSETTA_BR_CASE(13)
    default:
      return cudaErrorInvalidValue;
  }
#undef ROSETTA_BR_CASE
}

}  // namespace rosetta
