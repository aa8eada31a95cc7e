// LWE key switch on the tensor cores (tcgen05, accumulators in tensor memory).
//
// The key switch is the dense contraction of the path:
//   out[b][j] = [j = n] b'_b - sum_r d[b][r] KSK[r][j]      (mod 2^64)
// over r = (lev, i), the signed base-2^beta digits d of the extracted
// ciphertexts times the 64-bit key words.  It is made exact on bf16 tensor
// cores by cutting every key word into `limbs` unsigned limbs of 64/limbs
// bits, KSK = sum_t L_t 2^(t*64/limbs):  every digit (|d| <= 2^(beta-1)) and
// every limb is an integer that bf16 holds exactly, every product is exact in
// the fp32 accumulator, and every partial sum stays below 2^24 (checked on
// the host: 2^(beta-1) (2^(64/limbs) - 1) K < 2^24 with K = kN l), so the
// fp32 results are the exact integers C_t[b][j] = sum_r d[b][r] L_t[r][j] and
//   sum_r d KSK = sum_t C_t 2^(t*64/limbs)   (mod 2^64)
// is recombined in the epilogue.  Same words as keyswitch_kernel.
//
// Operands.  A = digits [batch x K] and B = limbs [K x limbs (n+1)] are both
// kept in global memory already cut into the tiles one MMA step consumes, in
// the no-swizzle K-major layout of the tensor cores (core matrices of 8 rows
// x 16 bytes; K-adjacent core matrices 128 B apart, 8-row groups 1024 B
// apart), so one bulk copy per tile brings it into shared memory.  K runs
// level-major (r = (lev-1) kN + i), so a 64-wide K step has one level.  The
// key's tiles are built once at upload, the digit tiles by ks_digits_kernel
// per call.
//
// Per CTA: a 128 x 256 output tile (128 ciphertexts x 256 limb columns =
// 256/limbs output words each), a 3-stage ring of 48 KB (A 16 KB + B 32 KB)
// filled by cp.async.bulk, one thread issuing tcgen05.mma (M = 128, N = 256,
// K = 16, four per step) into 256 columns of tensor memory, and four warps
// reading their 32 lanes back with tcgen05.ld for the recombination.  Every
// wait on an mbarrier gives up after about two seconds and sets the error
// flag; the CTA then skips its epilogue, waits (again bounded) for the copies
// it issued, and frees the tensor memory only when nothing it issued can
// still be in flight.
#include <stdint.h>

#include "dsmem.cuh"
#include "internal.h"

namespace rosetta {

namespace {

constexpr uint32_t TC_M = 128, TC_N = 256, TC_K = 64, TC_STAGES = 3, TC_THREADS = 128;
constexpr uint32_t A_TILE = TC_M * TC_K * 2;   // bytes
constexpr uint32_t B_TILE = TC_N * TC_K * 2;
constexpr uint32_t STAGE = A_TILE + B_TILE;
constexpr uint32_t TMEM_COLS = 256;
constexpr long long kWaitCycles = 4000000000ll;  // ~2 s at 2 GHz

// Element offset of (row, k) inside a tile of the no-swizzle K-major layout.
__host__ __device__ constexpr uint32_t tile_off(uint32_t row, uint32_t k) {
  return (((row >> 3) * (TC_K / 8) + (k >> 3)) << 6) + ((row & 7u) << 3) + (k & 7u);
}

__device__ __forceinline__ uint16_t bf16_of_int(int v) {
  // |v| <= 256: exact in bf16 (8 significant bits); the top half of the fp32 bits
  const float f = static_cast<float>(v);
  return static_cast<uint16_t>(__float_as_uint(f) >> 16);
}

// Shared-memory matrix descriptor: start address, leading (K) byte offset 128,
// stride (8-row) byte offset 1024, descriptor version 1, no swizzle.
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr) {
  return static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4) | (static_cast<uint64_t>(128u >> 4) << 16) |
         (static_cast<uint64_t>(1024u >> 4) << 32) | (1ull << 46);
}

// Instruction descriptor, kind::f16: D f32, A and B bf16, both K-major,
// N = 256, M = 128.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((TC_N >> 3) << 17) | ((TC_M >> 4) << 24);

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, long long limit = kWaitCycles) {
  const long long t0 = clock64();
  while (true) {
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\tselp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(bar), "r"(parity)
        : "memory");
    if (done) return true;
    if (clock64() - t0 > limit) return false;
  }
}

__device__ __forceinline__ void bulk_load(uint32_t dst, const void *src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "l"(src), "r"(bytes), "r"(bar)
               : "memory");
}

__device__ __forceinline__ void expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

__device__ __forceinline__ void mma_bf16(uint32_t tmem, uint64_t adesc, uint64_t bdesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem),
      "l"(adesc), "l"(bdesc), "r"(kIdesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}

// 32 consecutive fp32 columns of this thread's lane
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]), "=r"(v[8]),
        "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]), "=r"(v[16]),
        "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]),
        "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

}  // namespace

// Digit tiles: A[b][r] = digit lev of a'_i, r = (lev-1) kN + i, for one
// 128 x 64 tile per CTA (grid: k_steps x m_tiles), written 8 digits (16 B) at
// a time.  The balanced digits of the rounded value v are the plain base-B
// digits of v + sum_m (B/2) B^m minus B/2 (the carry rule of the
// decomposition, in closed form).
__global__ void __launch_bounds__(256) ks_digits_kernel(const uint64_t *__restrict__ big, uint16_t *__restrict__ a_tiles,
                                                        uint32_t batch, uint32_t kN, uint32_t base_log, uint32_t level,
                                                        uint32_t k_steps) {
  const uint32_t ks = blockIdx.x, mt = blockIdx.y;
  const uint32_t r0 = ks * TC_K;
  const uint32_t lev = r0 / kN + 1;  // 1 = most significant
  const uint32_t i0 = r0 % kN;
  const uint32_t bits = base_log * level;
  const uint64_t B = 1ull << base_log, Bmask = B - 1;
  uint64_t C = 0;
  for (uint32_t m = 0; m < level; ++m) C |= (B >> 1) << (m * base_log);
  const uint32_t sh = base_log * (level - lev);
  uint16_t *tile = a_tiles + (static_cast<size_t>(mt) * k_steps + ks) * (TC_M * TC_K);
  for (uint32_t item = threadIdx.x; item < TC_M * (TC_K / 8); item += blockDim.x) {
    const uint32_t row = item / (TC_K / 8), kg = item % (TC_K / 8);
    const uint32_t b = mt * TC_M + row;
    uint32_t packed[4] = {0u, 0u, 0u, 0u};
    if (b < batch) {
      const uint64_t *src = big + static_cast<size_t>(b) * (kN + 1) + i0 + kg * 8;
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const uint64_t a = src[e];
        uint64_t v = bits >= 64 ? a : (a + (1ull << (63 - bits))) >> (64 - bits);
        v += C;
        if (bits < 64) v &= (1ull << bits) - 1;
        const int d = static_cast<int>((v >> sh) & Bmask) - static_cast<int>(B >> 1);
        packed[e >> 1] |= static_cast<uint32_t>(bf16_of_int(d)) << (16 * (e & 1));
      }
    }
    *reinterpret_cast<uint4 *>(tile + tile_off(row, kg * 8)) = make_uint4(packed[0], packed[1], packed[2], packed[3]);
  }
}

// Limb tiles of the key: B[r][c] = limb t of KSK[i][lev-1][j], c = j limbs + t,
// zero beyond column n.  Grid: k_steps x n_tiles, once per key.
__global__ void __launch_bounds__(256) ks_limbs_kernel(const uint64_t *__restrict__ ksk, uint16_t *__restrict__ b_tiles,
                                                       uint32_t kN, uint32_t level, uint32_t n, uint32_t limbs,
                                                       uint32_t k_steps) {
  const uint32_t ks = blockIdx.x, nt = blockIdx.y;
  const uint32_t r0 = ks * TC_K;
  const uint32_t lev = r0 / kN + 1, i0 = r0 % kN;
  const uint32_t lbits = 64 / limbs;
  const uint64_t lmask = (1ull << lbits) - 1;
  uint16_t *tile = b_tiles + (static_cast<size_t>(nt) * k_steps + ks) * (TC_N * TC_K);
  for (uint32_t item = threadIdx.x; item < TC_N * (TC_K / 8); item += blockDim.x) {
    const uint32_t col = item / (TC_K / 8), kg = item % (TC_K / 8);
    const uint32_t c = nt * TC_N + col, j = c / limbs, t = c % limbs;
    uint32_t packed[4] = {0u, 0u, 0u, 0u};
    if (j <= n) {
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const uint32_t i = i0 + kg * 8 + e;
        const uint64_t w = ksk[(static_cast<size_t>(i) * level + (lev - 1)) * (n + 1) + j];
        packed[e >> 1] |= static_cast<uint32_t>(bf16_of_int(static_cast<int>((w >> (lbits * t)) & lmask)))
                          << (16 * (e & 1));
      }
    }
    *reinterpret_cast<uint4 *>(tile + tile_off(col, kg * 8)) = make_uint4(packed[0], packed[1], packed[2], packed[3]);
  }
}

template <uint32_t LIMBS>
__global__ void __launch_bounds__(TC_THREADS, 1) ks_tc_kernel(const KsTcArgs a) {
  extern __shared__ __align__(1024) unsigned char smem[];
  __shared__ __align__(8) uint64_t bars[2 * TC_STAGES + 1];  // full[s], empty[s], done
  __shared__ uint32_t tmem_slot;
  // set when a wait gave up: s_fail, a copy or an MMA slot never completed
  // (the accumulators are partial); s_unsafe, copies or MMAs this CTA issued
  // may still be in flight
  __shared__ uint32_t s_fail, s_unsafe;
  const uint32_t nt = blockIdx.x, mt = blockIdx.y;
  const uint32_t warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const uint32_t base = smem_addr(smem);
  const uint32_t bar0 = smem_addr(bars);
  auto full = [&](uint32_t s) { return bar0 + 8u * s; };
  auto empty = [&](uint32_t s) { return bar0 + 8u * (TC_STAGES + s); };
  const uint32_t done = bar0 + 8u * (2 * TC_STAGES);

  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(&tmem_slot)),
                 "r"(TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  if (threadIdx.x == 0) {
    s_fail = 0u;
    s_unsafe = 0u;
    for (uint32_t s = 0; s < 2 * TC_STAGES + 1; ++s) mbar_init(bar0 + 8u * s, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = tmem_slot;

  const uint32_t steps = a.k_steps;
  const uint16_t *atile = a.a_tiles + static_cast<size_t>(mt) * steps * (TC_M * TC_K);
  const uint16_t *btile = a.b_tiles + static_cast<size_t>(nt) * steps * (TC_N * TC_K);
  bool ok = true;
  if (warp == 0) {
    if (lane == 0) {
      auto issue = [&](uint32_t k, uint32_t slot) {
        expect_tx(full(slot), STAGE);
        bulk_load(base + slot * STAGE, atile + static_cast<size_t>(k) * (TC_M * TC_K), A_TILE, full(slot));
        bulk_load(base + slot * STAGE + A_TILE, btile + static_cast<size_t>(k) * (TC_N * TC_K), B_TILE, full(slot));
      };
      const uint32_t pre = steps < TC_STAGES ? steps : TC_STAGES;
      for (uint32_t k = 0; k < pre; ++k) issue(k, k);
      uint32_t issued = pre, consumed = 0;
      for (uint32_t k = 0; k < steps; ++k) {
        const uint32_t slot = k % TC_STAGES, par = (k / TC_STAGES) & 1u;
        if (!mbar_wait(full(slot), par)) {
          ok = false;
          break;
        }
        consumed = k + 1;
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t sa = base + slot * STAGE, sb = sa + A_TILE;
#pragma unroll
        for (uint32_t kk = 0; kk < TC_K / 16; ++kk)  // K = 16 per MMA: two core matrices, 256 B
          mma_bf16(tmem, smem_desc(sa + kk * 256u), smem_desc(sb + kk * 256u), (k | kk) != 0);
        mma_commit(empty(slot));
        if (k + TC_STAGES < steps) {
          if (!mbar_wait(empty(slot), par)) {  // the MMAs reading this slot are done
            ok = false;
            break;
          }
          issue(k + TC_STAGES, slot);
          ++issued;
        }
      }
      mma_commit(done);
      if (!ok) {
        atomicExch(a.err_flag, 2u);
        s_fail = 1u;
        // let the copies already issued land before the shared memory is released
        bool drained = true;
        for (uint32_t k = consumed; k < issued; ++k)
          drained = mbar_wait(full(k % TC_STAGES), (k / TC_STAGES) & 1u) && drained;
        if (!drained) s_unsafe = 1u;
      }
    }
    __syncwarp();
  }
  const bool fin = __all_sync(0xffffffffu, mbar_wait(done, 0));  // warp-uniform for tcgen05.ld
  if (!fin && lane == 0) {
    atomicExch(a.err_flag, 2u);
    s_unsafe = 1u;  // the MMAs may still be writing tensor memory
  }
  __syncthreads();
  const bool unsafe = s_unsafe != 0u, partial = s_fail != 0u;
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");

  if (!unsafe && !partial) {
    // epilogue: lane = ciphertext row of this warp's quarter of tensor memory
    const uint32_t row = warp * 32 + lane;
    const uint32_t b = mt * TC_M + row;
    constexpr uint32_t lbits = 64 / LIMBS;
    constexpr uint32_t per_chunk = 32 / LIMBS;  // output words per 32 columns
    const uint32_t n1 = a.n + 1;
    const uint64_t body = b < a.batch ? a.big[static_cast<size_t>(b) * (a.kN + 1) + a.kN] : 0;
#pragma unroll 1
    for (uint32_t q = 0; q < TC_N / 32; ++q) {
      uint32_t v[32];
      tmem_ld32(tmem + ((warp * 32u) << 16) + q * 32u, v);
#pragma unroll
      for (uint32_t jj = 0; jj < per_chunk; ++jj) {
        uint64_t s = 0;
#pragma unroll
        for (uint32_t t = 0; t < LIMBS; ++t) {
          const int64_t c = __float2int_rn(__uint_as_float(v[jj * LIMBS + t]));
          s += static_cast<uint64_t>(c) << (lbits * t);
        }
        const uint32_t j = (nt * TC_N + q * 32) / LIMBS + jj;
        if (b < a.batch && j < n1) a.out[static_cast<size_t>(b) * n1 + j] = (j == a.n ? body : 0ull) - s;
      }
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  // After a wait that gave up with work still in flight nothing is safe: the
  // tensor memory is left allocated rather than handed to another CTA while
  // an MMA may still write it, the outputs are not written, and the error
  // flag reports TIMEOUT.  The CUDA context must then be destroyed.
  if (warp == 0 && !unsafe)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TMEM_COLS) : "memory");
}

// Self-test of the bounded-wait path: one thread waits on an mbarrier that
// nothing completes, gives up after `limit` cycles and reports it through the
// error flag exactly as ks_tc_kernel does.
__global__ void wait_selftest_kernel(uint32_t *err_flag, long long limit) {
  __shared__ __align__(8) uint64_t bar;
  const uint32_t b = smem_addr(&bar);
  mbar_init(b, 1);
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  if (!mbar_wait(b, 0, limit)) atomicExch(err_flag, 2u);
}

cudaError_t launch_wait_selftest(uint32_t *err_flag, uint32_t limit_us, cudaStream_t s) {
  wait_selftest_kernel<<<1, 1, 0, s>>>(err_flag, static_cast<long long>(limit_us) * 2000);  // ~2 GHz
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------- host side

uint32_t ks_tc_limbs(uint32_t kN, uint32_t level, uint32_t base_log) {
  if (base_log > 8 || (static_cast<uint64_t>(kN) * level) % TC_K != 0) return 0;
  const double K = static_cast<double>(kN) * level, dmax = static_cast<double>(1u << (base_log - 1));
  for (uint32_t limbs : {8u, 16u})
    if (dmax * static_cast<double>((1ull << (64 / limbs)) - 1) * K < 16777216.0) return limbs;
  return 0;
}

size_t ks_tc_b_words16(uint32_t kN, uint32_t level, uint32_t n, uint32_t limbs) {
  const size_t k_steps = static_cast<size_t>(kN) * level / TC_K;
  const size_t n_tiles = (static_cast<size_t>(n + 1) * limbs + TC_N - 1) / TC_N;
  return n_tiles * k_steps * TC_N * TC_K;
}

size_t ks_tc_a_words16(uint32_t batch, uint32_t kN, uint32_t level) {
  const size_t k_steps = static_cast<size_t>(kN) * level / TC_K;
  const size_t m_tiles = (batch + TC_M - 1) / TC_M;
  return m_tiles * k_steps * TC_M * TC_K;
}

cudaError_t launch_ks_limbs(const uint64_t *ksk, uint16_t *b_tiles, uint32_t kN, uint32_t level, uint32_t n,
                            uint32_t limbs, cudaStream_t s) {
  const uint32_t k_steps = kN * level / TC_K;
  const uint32_t n_tiles = ((n + 1) * limbs + TC_N - 1) / TC_N;
  ks_limbs_kernel<<<dim3(k_steps, n_tiles), 256, 0, s>>>(ksk, b_tiles, kN, level, n, limbs, k_steps);
  return cudaGetLastError();
}

cudaError_t launch_keyswitch_tc(const KsTcArgs &a, uint32_t base_log, uint32_t level, cudaStream_t s) {
  const uint32_t m_tiles = (a.batch + TC_M - 1) / TC_M;
  const uint32_t n_tiles = ((a.n + 1) * a.limbs + TC_N - 1) / TC_N;
  ks_digits_kernel<<<dim3(a.k_steps, m_tiles), 256, 0, s>>>(a.big, const_cast<uint16_t *>(a.a_tiles), a.batch, a.kN,
                                                             base_log, level, a.k_steps);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int smem = static_cast<int>(TC_STAGES * STAGE);
  auto kern = a.limbs == 8 ? ks_tc_kernel<8> : ks_tc_kernel<16>;
  e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  kern<<<dim3(n_tiles, m_tiles), TC_THREADS, smem, s>>>(a);
  return cudaGetLastError();
}

}  // namespace rosetta
