// Internal declarations of librosetta shared by the host API and the kernels.
#pragma once
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace rosetta {

// Four NTT primes p = c * 2^14 + 1 in (2^28 - 2^18, 2^28): 2N | p - 1 for every
// N <= 8192, 16p < 2^32 leaves room for lazily reduced residues, and their
// product M > 2^111.99 exceeds twice the largest exact integer value of an
// external-product coefficient, (k+1) l N 2^(beta-1) 2^63, for every
// parameter set the library accepts (checked at context creation).
constexpr int kPrimes = 4;
constexpr uint32_t kPrimeList[kPrimes] = {268369921u, 268271617u, 268238849u, 268189697u};

// Three NTT primes p = c * 2^14 + 1 in (2^31 - 2^19, 2^31), product
// M > 2^92.999: the blind rotation's prime set for the parameter sets whose
// external-product bound stays below 0.45 M (N = 4096 with (k+1) l 2^beta up
// to 2^17, e.g. l = 2, beta = 15; N = 8192 up to 2^16.8, e.g. l = 3,
// beta = 14).  No lazy headroom (4p > 2^32): residues are kept in [0, 2p).
constexpr int kPrimes31 = 3;
constexpr uint32_t kPrime31List[kPrimes31] = {2147352577u, 2147205121u, 2147074049u};

struct PrimeConsts {
  uint32_t p;
  uint32_t p_inv;     // p^{-1} mod 2^32 (Montgomery reduction)
  uint32_t crt_c;     // N^{-1} * (M/p)^{-1} mod p (folded into the transformed keys)
  uint32_t crt_cs;    // Shoup companion of crt_c
  uint32_t key_scale;    // 2^32 crt_c mod p: Montgomery form times the CRT factor
  uint32_t key_scale_s;  // Shoup companion of key_scale
  uint64_t Mp_mod64;  // (M / p) mod 2^64
};

struct CrtConsts {
  PrimeConsts pr[kPrimes];
  uint64_t M_mod64;   // M mod 2^64
};

struct BrArgs {
  const uint64_t *lwe_in;   // [batch][n+1]
  const uint64_t *lut;      // [num_luts][2^p]; ignored when glwe_in is set
  uint64_t *lwe_big_out;    // [batch][N+1] extracted LWEs (k = 1), or
  uint64_t *glwe_out;       // [batch][2][N] rotated accumulators (when set)
  const uint32_t *lut_index;  // [batch] LUT of each ciphertext, or null (LUT 0)
  const uint64_t *glwe_in;  // [batch][2][N] GLWE test polynomials, or null
  uint32_t *err_flag;       // set to 1 when a LUT index is out of range
  const uint32_t *bsk;      // transform domain [n][prime][2l][2][N]
  size_t bsk_words;         // words of bsk (checked by ROSETTA_DEBUG builds; 0: unchecked)
  const uint2 *tw;          // [prime][N] (W, Shoup companion)
  uint32_t n, level, base_log, msg_bits, batch, num_luts;
  uint32_t primes;          // kPrimes (bsk, tw, cc over the 28-bit set) or kPrimes31
  CrtConsts cc;
};

struct KsArgs {
  const uint64_t *big;      // [batch][kN+1]
  uint64_t *out;            // [batch][n+1]
  const uint64_t *ksk;      // [kN][l_ks][n+1]
  const uint64_t *corr;     // [n+1]: (B/2) * sum over KSK rows
  uint32_t batch, kN, n, base_log, level;
};

// Tensor-core key switch: digit and limb tiles in the MMA layout.
struct KsTcArgs {
  const uint16_t *a_tiles;  // [m_tiles][k_steps][128 x 64] bf16 digits
  const uint16_t *b_tiles;  // [n_tiles][k_steps][256 x 64] bf16 key limbs
  const uint64_t *big;      // [batch][kN+1]
  uint64_t *out;            // [batch][n+1]
  uint32_t *err_flag;       // set to 2 when a wait gives up
  uint32_t batch, kN, n, k_steps, limbs;
};

struct TraceArgs {
  const uint64_t *glwe_in;  // [batch][2][N]
  uint64_t *glwe_out;       // [batch][2][N]
  const uint32_t *keys;     // transform domain [steps][prime][rows][2][N]
  const uint64_t *plain_add;  // [N] added to the body (plaintext-multiply mode), or null
  const uint2 *tw;          // [prime][N]
  uint32_t base_log, level, batch;  // level = rows of a key (trace); 2 x gadget levels (multiply)
  CrtConsts cc;
};

// Cluster placement of a blind-rotation launch of `ctas` CTAs: packed onto
// the SMs with room (load-balancing) once the launch fills every CTA slot of
// the GPU at least once, spread over the SMs below that.  Measured on GB300:
// load-balancing is 2-2.5 % faster for full batches and 5.6 % slower for a
// partial wave (256 CTAs of the standard set).
template <typename K>
inline cudaClusterSchedulingPolicy br_cluster_policy(K kern, int threads, size_t smem, size_t ctas) {
  int dev = 0, sms = 0, per_sm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, threads, smem) != cudaSuccess) {
    cudaGetLastError();  // the query's own error; the launch decides the rest
    return cudaClusterSchedulingPolicySpread;
  }
  return ctas >= static_cast<size_t>(sms) * static_cast<size_t>(per_sm) ? cudaClusterSchedulingPolicyLoadBalancing
                                                                        : cudaClusterSchedulingPolicySpread;
}

// host-side tables (tables.cu): twiddles and CRT constants of the 28-bit set
// (primes = kPrimes) or of the 31-bit set (primes = kPrimes31)
bool build_tables(uint32_t logN, uint32_t primes, uint2 *tw_host /*[primes][N]*/, CrtConsts *cc);

// launchers; return cudaSuccess or the launch error
size_t br_smem_bytes(uint32_t logN, uint32_t level, uint32_t n, bool dig16);
// a.primes selects the kernel: the four-prime one or the three-prime one
cudaError_t launch_blind_rotate(const BrArgs &a, uint32_t logN, bool dig16, cudaStream_t s);
// three-prime kernel (blind_rotate3.cu): 16-bit digits, compiled ring sizes and levels only
bool br3_supported(uint32_t logN, uint32_t level, bool dig16);
size_t br3_smem_bytes(uint32_t logN, uint32_t level, uint32_t n);
cudaError_t launch_blind_rotate3(const BrArgs &a, uint32_t logN, cudaStream_t s);
cudaError_t launch_bsk_transform(const uint64_t *raw, uint32_t *out, const uint2 *tw, const CrtConsts &cc,
                                 uint32_t logN, uint32_t n, uint32_t level, uint32_t primes, cudaStream_t s);
cudaError_t launch_keyswitch(const KsArgs &a, cudaStream_t s);
// transform `count` raw keys [count][rows][2][N] to [count][prime][rows][2][N]
// over the 28-bit set (primes = kPrimes) or the 31-bit set (kPrimes31)
cudaError_t launch_key_transform(const uint64_t *raw, uint32_t *out, const uint2 *tw, const CrtConsts &cc,
                                 uint32_t logN, uint32_t count, uint32_t rows, cudaStream_t s,
                                 uint32_t primes = kPrimes);
size_t trace_smem_bytes(uint32_t logN, uint32_t level);
cudaError_t launch_trace(const TraceArgs &a, uint32_t logN, cudaStream_t s);
cudaError_t launch_plaintext_mul(const TraceArgs &a, uint32_t logN, cudaStream_t s);
cudaError_t launch_monomial_acc(uint64_t *R, const uint64_t *r, uint32_t count, uint32_t logN, uint32_t e, bool first,
                                cudaStream_t s);
uint32_t ks_tc_limbs(uint32_t kN, uint32_t level, uint32_t base_log);  // 8, 16, or 0 (not exact)
size_t ks_tc_b_words16(uint32_t kN, uint32_t level, uint32_t n, uint32_t limbs);
size_t ks_tc_a_words16(uint32_t batch, uint32_t kN, uint32_t level);
cudaError_t launch_ks_limbs(const uint64_t *ksk, uint16_t *b_tiles, uint32_t kN, uint32_t level, uint32_t n,
                            uint32_t limbs, cudaStream_t s);
cudaError_t launch_keyswitch_tc(const KsTcArgs &a, uint32_t base_log, uint32_t level, cudaStream_t s);
cudaError_t launch_wait_selftest(uint32_t *err_flag, uint32_t limit_us, cudaStream_t s);
cudaError_t launch_ksk_corr(const uint64_t *ksk, uint64_t *corr, uint32_t rows, uint32_t n, uint32_t base_log,
                            cudaStream_t s);

}  // namespace rosetta
