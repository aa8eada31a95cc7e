// Blind rotation over three NTT primes near 2^31, one thread-block cluster of
// three CTAs per ciphertext, for the parameter sets whose external-product
// coefficients stay below 0.45 M3 in magnitude (M3 > 2^92.999 the product of
// the three primes; checked at context creation).
//
// Same construction and step structure as the four-prime kernel
// (blind_rotate.cu; Background, "TFHE Scheme", PBS): the accumulator starts
// as X^{-b~} times the test polynomial and every CMux step adds
// BSK_i (x) (X^{a~_i} ACC - ACC), the external product computed exactly with
// negacyclic NTTs per prime and an explicit CRT.  What differs:
//   * prime arithmetic: the primes lie in (2^31 - 2^19, 2^31), so a residue
//     has no room to grow lazily (4p > 2^32); every value of the transforms
//     stays in [0, 2p) (the P31 butterflies of ntt.cuh), forward outputs are
//     brought below p before the multiply-accumulate, and the CRT quotient is
//     estimated against 2^31;
//   * ownership: the E = 8 first-pass slots of every thread are split 3/3/2
//     over the three CTAs, so CTA o owns the coefficients
//     [S_o N/8, S_{o+1} N/8) of both components, S = (0, 3, 6, 8), and holds
//     them as acc[component][slot h][thread tau];
//   * the residue exchange: a prime-CTA keeps the residues of its own slots in
//     registers across the cluster barrier (its threads are their owners) and
//     leaves every other owner's slots, one packed group per thread, in its
//     own exchange buffer, from which the owners read them in phase 3.
// Every cross-CTA read follows a write to the writer's own shared memory, so
// the step's barriers order shared memory only (cluster_sync_shared).
// Per ciphertext and step the cluster runs 3 (l + 1) x 2 transforms instead
// of 4 (l + 1) x 2; a butterfly is seven instructions instead of five and,
// measured alone, about 15 % slower.
#include <cooperative_groups.h>

#include "check.cuh"
#include "dsmem.cuh"
#include "internal.h"
#include "ntt.cuh"

namespace rosetta {
namespace cg = cooperative_groups;

namespace {

// first owned first-pass slot of CTA o (o = 3: the end)
__host__ __device__ constexpr uint32_t own_s0(int o) { return o == 0 ? 0u : (o == 1 ? 3u : (o == 2 ? 6u : 8u)); }

// owner of first-pass slot q < 8: 0, 0, 0, 1, 1, 1, 2, 2 (two bits per slot)
__device__ __forceinline__ uint32_t slot_owner(uint32_t q) { return (0xA540u >> (2u * q)) & 3u; }

template <int LOGN>
struct Br3Shape {
  static constexpr int N = 1 << LOGN;
  static constexpr int E = 8;
  static constexpr int T = N / E;  // threads per CTA
  static constexpr int LOG_T = LOGN - 3;
  // resident CTAs per SM the register allocation must allow (2 x 92-98 KB of
  // shared memory at N = 4096, 1 x 198 KB at 8192)
  static constexpr int MIN_CTAS = LOGN <= 12 ? 2 : 1;
  // exchange buffer words: N + N/8 for the transforms, extended to 12 T so
  // that it holds the outgoing residues afterwards
  static constexpr int XB_WORDS = 12 * T;
};

__device__ __forceinline__ uint32_t pack16(int32_t lo, int32_t hi) {
  return (static_cast<uint32_t>(lo) & 0xFFFFu) | (static_cast<uint32_t>(hi) << 16);
}
__device__ __forceinline__ int32_t lo16(uint32_t w) { return static_cast<int16_t>(w & 0xFFFFu); }
__device__ __forceinline__ int32_t hi16(uint32_t w) { return static_cast<int16_t>(w >> 16); }

}  // namespace

// Shared memory, in this order (16-byte aligned pieces):
//   tw    uint2  [N]           twiddles of prime `rank`
//   acc   uint64 [2][3][T]     owned accumulator words (component, slot, thread)
//   xb    uint32 [12 T]        transform exchange buffer (N + N/8 words); after the
//                              inverse transforms the outgoing residues: [2 other
//                              owners][T][4] (slots 0, 1 of both components), then
//                              [2][T][2] (slot 2, owners 0 and 1)
//   dig8  uint32 [l][T][2]     16-bit digits of each row pair: slots 0, 1 of both rows
//   dig4  uint32 [l][T]        slot 2 of both rows (owners 0 and 1)
//   atil  uint16 [n+1]         switched mask and body
size_t br3_smem_bytes(uint32_t logN, uint32_t level, uint32_t n) {
  const size_t N = size_t(1) << logN, T = N / 8;
  size_t b = N * sizeof(uint2) + 6 * T * sizeof(uint64_t) + (12 * T + 3 * level * T) * sizeof(uint32_t) +
             (n + 1) * sizeof(uint16_t);
  return (b + 15) & ~size_t(15);
}

template <int LOGN, int LEV>
__global__ void __launch_bounds__(Br3Shape<LOGN>::T, Br3Shape<LOGN>::MIN_CTAS) blind_rotate3_kernel(const BrArgs a) {
  using B = Br3Shape<LOGN>;
  using S = NttShape<LOGN, 8>;
  constexpr uint32_t N = B::N, T = B::T, TWO_N = 2 * N;
  constexpr int E = B::E;
  constexpr uint32_t L = LEV;  // gadget levels: 2 L rows, L row pairs

  cg::cluster_group cluster = cg::this_cluster();
  const uint32_t rank = cluster.block_rank();
  const uint32_t ct = blockIdx.x / 3;
  const uint32_t tau = threadIdx.x;
  if (!dbg_ok(ct < a.batch, a.err_flag)) return;  // the whole cluster shares ct

  extern __shared__ __align__(16) unsigned char smem[];
  static_assert(B::XB_WORDS >= S::XB_WORDS, "exchange buffer");
  uint2 *tw = reinterpret_cast<uint2 *>(smem);
  uint64_t *acc = reinterpret_cast<uint64_t *>(tw + N);
  uint32_t *xb = reinterpret_cast<uint32_t *>(acc + 6 * T);
  uint32_t *dig8 = xb + B::XB_WORDS;
  uint32_t *dig4 = dig8 + L * T * 2;
  uint16_t *atil = reinterpret_cast<uint16_t *>(dig4 + L * T);

  const uint32_t p = a.cc.pr[rank].p;
  const uint32_t p_inv = a.cc.pr[rank].p_inv;
  const uint32_t s0 = 3 * rank;   // first owned slot
  const bool three = rank < 2;    // owners 0 and 1 hold a third slot

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
      for (int c = 0; c < 2; ++c)
#pragma unroll
        for (int h = 0; h < 3; ++h) {
          if (h == 2 && !three) continue;
          const uint32_t j = tau + (s0 + h) * T;
          const uint32_t e = (j + btil) & (TWO_N - 1);
          const uint64_t v = gin[c * N + (e & (N - 1))];
          acc[(c * 3 + h) * T + tau] = (e >= N) ? 0ull - v : v;
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
      const uint32_t box = N >> a.msg_bits, hb = box >> 1;
#pragma unroll
      for (int h = 0; h < 3; ++h) {
        if (h == 2 && !three) continue;
        const uint32_t j = tau + (s0 + h) * T;
        acc[h * T + tau] = 0;
        // (X^{2N - b~} v)[j] = +-v[t], t = (j + b~) mod 2N folded into [0, N)
        const uint32_t e = (j + btil) & (TWO_N - 1);
        const uint32_t t = e & (N - 1);
        const uint64_t v = (t < N - hb) ? lut[(t + hb) / box] : (0ull - lut[0]);
        acc[(3 + h) * T + tau] = (e >= N) ? 0ull - v : v;
      }
    }
  }
  cluster.sync();

  const uint32_t acc_s = smem_addr(acc), dig8_s = smem_addr(dig8), dig4_s = smem_addr(dig4);
  const uint32_t xb_s = smem_addr(xb);
  const uint32_t bits = a.base_log * L;
  const uint64_t Bmask = (1ull << a.base_log) - 1;
  const uint64_t Bhalf = 1ull << (a.base_log - 1);
  const uint64_t round_add = bits >= 64 ? 0 : (1ull << (63 - bits));
  const uint32_t round_sh = bits >= 64 ? 0 : 64 - bits;

  for (uint32_t i = 0; i < a.n; ++i) {
    const uint32_t at = atil[i];
    if (at == 0) continue;  // X^0 ACC - ACC = 0: the step adds nothing

    // ---- phase 1: rotated difference and gadget digits of the owned slots ----
    // (X^a P)[j] = +-P[(j - a) mod 2N]: the source of slot (c, h) is slot
    // qs = e / T of thread e mod T (the same thread for every slot), held by
    // owner slot_owner(qs).  At N = 4096: slots 0 and 1 of both components
    // first (they complete every 8-byte digit group), then slot 2 (the 4-byte
    // groups; owners 0 and 1 only), which keeps fewer values live (no spills
    // with two levels; measured 1.9 % faster than the other order).  At
    // N = 8192: one component at a time, a row pair's digits stored as soon as
    // complete (row r = c l + lev, pair r / 2; measured 1.4 % faster there).
    if constexpr (LOGN <= 12) {
#pragma unroll
      for (int hg = 0; hg < 2; ++hg) {
        if (hg == 1 && !three) break;
        constexpr int NS_MAX = 2;
        const int h0 = hg == 0 ? 0 : 2, ns = hg == 0 ? 2 : 1;
        int32_t g[L][2][NS_MAX];  // [row pair][row parity][slot of the group]
        uint64_t v[2][NS_MAX];
#pragma unroll
        for (int c = 0; c < 2; ++c)
#pragma unroll
          for (int k = 0; k < NS_MAX; ++k) {
            if (k >= ns) continue;
            const uint32_t j = tau + (s0 + h0 + k) * T;
            const uint32_t e = (j + TWO_N - at) & (N - 1);
            const uint32_t qs = e >> B::LOG_T, os = slot_owner(qs);
            v[c][k] = dsmem_ld_u64(dsmem_map(acc_s + ((c * 3 + (qs - 3 * os)) * T + (e & (T - 1))) * 8u, os));
          }
#pragma unroll
        for (int c = 0; c < 2; ++c)
#pragma unroll
          for (int k = 0; k < NS_MAX; ++k) {
            if (k >= ns) continue;
            const int h = h0 + k;
            const uint32_t j = tau + (s0 + h) * T;
            const bool neg = ((j + TWO_N - at) & (TWO_N - 1)) >= N;
            const uint64_t diff = (neg ? 0ull - v[c][k] : v[c][k]) - acc[(c * 3 + h) * T + tau];
            uint64_t cv = bits >= 64 ? diff : (diff + round_add) >> round_sh;
#pragma unroll
            for (int l = static_cast<int>(L) - 1; l >= 0; --l) {
              const uint64_t d = cv & Bmask;
              cv >>= a.base_log;
              int32_t ds = static_cast<int32_t>(d);
              if (d >= Bhalf) {
                ds -= static_cast<int32_t>(Bmask + 1);
                cv += 1;
              }
              const int r = c * static_cast<int>(L) + l;
              g[r >> 1][r & 1][k] = ds;
            }
          }
#pragma unroll
        for (uint32_t P = 0; P < L; ++P) {
          if (hg == 0)
            *reinterpret_cast<uint2 *>(dig8 + (P * T + tau) * 2) =
                make_uint2(pack16(g[P][0][0], g[P][0][1]), pack16(g[P][1][0], g[P][1][1]));
          else
            dig4[P * T + tau] = pack16(g[P][0][0], g[P][1][0]);
        }
      }
    } else {
      int32_t g[L][2][3];  // [row pair][row parity][slot]
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        uint64_t v[3];
#pragma unroll
        for (int h = 0; h < 3; ++h) {
          if (h == 2 && !three) continue;
          const uint32_t j = tau + (s0 + h) * T;
          const uint32_t e = (j + TWO_N - at) & (N - 1);
          const uint32_t qs = e >> B::LOG_T, os = slot_owner(qs);
          v[h] = dsmem_ld_u64(dsmem_map(acc_s + ((c * 3 + (qs - 3 * os)) * T + (e & (T - 1))) * 8u, os));
        }
#pragma unroll
        for (int h = 0; h < 3; ++h) {
          if (h == 2 && !three) continue;
          const uint32_t j = tau + (s0 + h) * T;
          const bool neg = ((j + TWO_N - at) & (TWO_N - 1)) >= N;
          const uint64_t diff = (neg ? 0ull - v[h] : v[h]) - acc[(c * 3 + h) * T + tau];
          uint64_t cv = bits >= 64 ? diff : (diff + round_add) >> round_sh;
#pragma unroll
          for (int l = static_cast<int>(L) - 1; l >= 0; --l) {
            const uint64_t d = cv & Bmask;
            cv >>= a.base_log;
            int32_t ds = static_cast<int32_t>(d);
            if (d >= Bhalf) {
              ds -= static_cast<int32_t>(Bmask + 1);
              cv += 1;
            }
            const int r = c * static_cast<int>(L) + l;
            g[r >> 1][r & 1][h] = ds;
          }
        }
#pragma unroll
        for (int P = 0; P < static_cast<int>(L); ++P) {
          if ((2 * P + 1) / static_cast<int>(L) != c) continue;  // completed by this component
          *reinterpret_cast<uint2 *>(dig8 + (P * T + tau) * 2) =
              make_uint2(pack16(g[P][0][0], g[P][0][1]), pack16(g[P][1][0], g[P][1][1]));
          if (three) dig4[P * T + tau] = pack16(g[P][0][2], g[P][1][2]);
        }
      }
    }
    cluster_sync_shared();

    // ---- phase 2: transforms and pointwise products for prime `rank` ----
    uint32_t oh[2][E];
    const size_t kblk = static_cast<size_t>(2 * L) * 2 * N;  // words of one step's key block per prime
    const uint32_t *gbase = a.bsk + (static_cast<size_t>(i) * kPrimes31 + rank) * kblk;
    const bool key_ok = dbg_ok(
        a.bsk_words == 0 || (static_cast<size_t>(i) * kPrimes31 + rank + 1) * kblk <= a.bsk_words, a.err_flag);
#pragma unroll 1
    for (uint32_t P = 0; P < L; ++P) {
      // first-pass slot q of thread tau is coefficient tau + q N/8: slots
      // [own_s0(o), own_s0(o+1)) come from owner o, two 16-bit digits of each
      // of the pair's rows per packed word
      uint32_t x[2][E];
#pragma unroll
      for (int o = 0; o < 3; ++o) {
        const uint32_t q = own_s0(o);
        const uint2 w = dsmem_ld_v2_u32(dsmem_map(dig8_s + (P * T + tau) * 8u, o));
        x[0][q] = static_cast<uint32_t>(lo16(w.x)) + p;  // (0, 2p)
        x[0][q + 1] = static_cast<uint32_t>(hi16(w.x)) + p;
        x[1][q] = static_cast<uint32_t>(lo16(w.y)) + p;
        x[1][q + 1] = static_cast<uint32_t>(hi16(w.y)) + p;
        if (o < 2) {
          const uint32_t w4 = dsmem_ld_u32(dsmem_map(dig4_s + (P * T + tau) * 4u, o));
          x[0][q + 2] = static_cast<uint32_t>(lo16(w4)) + p;
          x[1][q + 2] = static_cast<uint32_t>(hi16(w4)) + p;
        }
      }
      ntt_forward<LOGN, E, 2, 1, true>(x, tw, xb, tau, p);  // outputs in [0, 2p)
      // below p, so that a row pair's two products sum below 2 p^2 < p 2^32
#pragma unroll
      for (int pp = 0; pp < 2; ++pp)
#pragma unroll
        for (int e = 0; e < E; ++e) x[pp][e] = cond_sub(x[pp][e], p);
      // BSK_i words of this prime for rows 2P, 2P+1, E per thread and
      // component, contiguous across the CTA (16-byte loads)
      const uint4 *gk = reinterpret_cast<const uint4 *>(gbase + static_cast<size_t>(2 * P) * 2 * N + E * tau);
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        uint32_t ga[E], gb[E];
#pragma unroll
        for (int k = 0; k < E / 4; ++k) {
          const uint4 va = key_ok ? __ldg(gk + (c * N) / 4 + k) : make_uint4(0u, 0u, 0u, 0u);
          const uint4 vb = key_ok ? __ldg(gk + ((2 + c) * N) / 4 + k) : make_uint4(0u, 0u, 0u, 0u);
          ga[4 * k] = va.x; ga[4 * k + 1] = va.y; ga[4 * k + 2] = va.z; ga[4 * k + 3] = va.w;
          gb[4 * k] = vb.x; gb[4 * k + 1] = vb.y; gb[4 * k + 2] = vb.z; gb[4 * k + 3] = vb.w;
        }
#pragma unroll
        for (int e = 0; e < E; ++e) {
          const uint64_t prod = static_cast<uint64_t>(x[0][e]) * ga[e] + static_cast<uint64_t>(x[1][e]) * gb[e];
          const uint32_t rr = redc(prod, p, p_inv);  // (0, 2p)
          oh[c][e] = (P == 0) ? rr : cond_sub(oh[c][e], p) + cond_sub(rr, p);  // [0, 2p)
        }
      }
    }
    ntt_inverse<LOGN, E, 2, 1, true>(oh, tw, xb, tau, p);  // outputs in [0, 2p)
    // CRT-scaled residues (the keys carry the CRT factor): one packed group
    // per other owner, left in this CTA's exchange buffer (once every thread
    // has finished the transforms' last exchange) at the owner's index among
    // the other two; the own slots stay in registers
    __syncthreads();
#pragma unroll
    for (int o = 0; o < 3; ++o) {
      if (static_cast<uint32_t>(o) == rank) continue;
      const uint32_t q = own_s0(o);
      const uint32_t oi = static_cast<uint32_t>(o) < rank ? o : o - 1;  // owner o among the other two
      *reinterpret_cast<uint4 *>(xb + (oi * T + tau) * 4) = make_uint4(oh[0][q], oh[0][q + 1], oh[1][q], oh[1][q + 1]);
      if (o < 2) *reinterpret_cast<uint2 *>(xb + 8 * T + (oi * T + tau) * 2) = make_uint2(oh[0][q + 2], oh[1][q + 2]);
    }
    uint32_t yo[2][3];
#pragma unroll
    for (int c = 0; c < 2; ++c) {
      yo[c][0] = rank == 0 ? oh[c][0] : (rank == 1 ? oh[c][3] : oh[c][6]);
      yo[c][1] = rank == 0 ? oh[c][1] : (rank == 1 ? oh[c][4] : oh[c][7]);
      yo[c][2] = rank == 0 ? oh[c][2] : oh[c][5];
    }
    cluster_sync_shared();

    // ---- phase 3: explicit CRT of the owned slots, accumulate ----
    {
      // the two other primes (producers), and this owner's index among the
      // other two owners of each; their residue groups read remotely
      const uint32_t q_r0 = rank == 0 ? 1u : 0u, q_r1 = rank == 2 ? 1u : 2u;
      const uint32_t oa = rank < q_r0 ? rank : rank - 1, ob = rank < q_r1 ? rank : rank - 1;
      const uint32_t pa = dsmem_map(xb_s, q_r0), pb = dsmem_map(xb_s, q_r1);
      const uint4 ra = dsmem_ld_v4_u32(pa + (oa * T + tau) * 16u);
      const uint4 rb = dsmem_ld_v4_u32(pb + (ob * T + tau) * 16u);
      uint2 sa = make_uint2(0u, 0u), sb = make_uint2(0u, 0u);
      if (three) {
        sa = dsmem_ld_v2_u32(pa + 32u * T + (oa * T + tau) * 8u);
        sb = dsmem_ld_v2_u32(pb + 32u * T + (ob * T + tau) * 8u);
      }
      const uint32_t y1[2][3] = {{ra.x, ra.y, sa.x}, {ra.z, ra.w, sa.y}};
      const uint32_t y2[2][3] = {{rb.x, rb.y, sb.x}, {rb.z, rb.w, sb.y}};
      const uint64_t m0 = a.cc.pr[rank].Mp_mod64, m1 = a.cc.pr[q_r0].Mp_mod64, m2 = a.cc.pr[q_r1].Mp_mod64;
#pragma unroll
      for (int c = 0; c < 2; ++c)
#pragma unroll
        for (int h = 0; h < 3; ++h) {
          if (h == 2 && !three) continue;
          const uint32_t ya = yo[c][h], yb = y1[c][h], yc = y2[c][h];
          const uint64_t s = static_cast<uint64_t>(ya) * m0 + static_cast<uint64_t>(yb) * m1 +
                             static_cast<uint64_t>(yc) * m2;
          const uint32_t u = crt_quotient31((ya >> 3) + (yb >> 3) + (yc >> 3));
          acc[(c * 3 + h) * T + tau] += s - static_cast<uint64_t>(u) * a.cc.M_mod64;
        }
    }
    cluster_sync_shared();
  }

  if (a.glwe_out) {
    // ---- the rotated accumulator itself ----
    uint64_t *gout = a.glwe_out + static_cast<size_t>(ct) * 2 * N;
#pragma unroll
    for (int c = 0; c < 2; ++c)
#pragma unroll
      for (int h = 0; h < 3; ++h) {
        if (h == 2 && !three) continue;
        gout[c * N + tau + (s0 + h) * T] = acc[(c * 3 + h) * T + tau];
      }
  } else {
    // ---- sample extraction of the constant coefficient ----
    uint64_t *out = a.lwe_big_out + static_cast<size_t>(ct) * (N + 1);
#pragma unroll
    for (int h = 0; h < 3; ++h) {
      if (h == 2 && !three) continue;
      const uint32_t j = tau + (s0 + h) * T;
      const uint64_t w = acc[h * T + tau];
      out[j == 0 ? 0 : N - j] = (j == 0) ? w : 0ull - w;
      if (j == 0) out[N] = acc[3 * T + tau];
    }
  }
  cluster.sync();
}

// Compiled: N = 4096 and 8192 with one to three levels.  The context also
// checks that the CTAs fit an SM as densely as the four-prime kernel's.
bool br3_supported(uint32_t logN, uint32_t level, bool dig16) {
  return dig16 && (logN == 12 || logN == 13) && level >= 1 && level <= 3;
}

template <int LOGN, int LEV>
static cudaError_t launch_br3_t(const BrArgs &a, cudaStream_t s) {
  auto kern = blind_rotate3_kernel<LOGN, LEV>;
  const size_t smem = br3_smem_bytes(LOGN, LEV, a.n);
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(3 * a.batch, 1, 1);
  cfg.blockDim = dim3(Br3Shape<LOGN>::T, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 3;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeClusterSchedulingPolicyPreference;
  attr[1].val.clusterSchedulingPolicyPreference = br_cluster_policy(kern, Br3Shape<LOGN>::T, smem, cfg.gridDim.x);
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, a);
}

cudaError_t launch_blind_rotate3(const BrArgs &a, uint32_t logN, cudaStream_t s) {
  if (a.primes != kPrimes31 || !br3_supported(logN, a.level, true)) return cudaErrorInvalidValue;
  if (logN == 12) {
    switch (a.level) {
      case 1: return launch_br3_t<12, 1>(a, s);
      case 2: return launch_br3_t<12, 2>(a, s);
      default: return launch_br3_t<12, 3>(a, s);
    }
  }
  switch (a.level) {
    case 1: return launch_br3_t<13, 1>(a, s);
    case 2: return launch_br3_t<13, 2>(a, s);
    default: return launch_br3_t<13, 3>(a, s);
  }
}

}  // namespace rosetta
