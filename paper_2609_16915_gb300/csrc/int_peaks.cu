// Integer issue-rate microbenchmarks: how many 32-bit integer operations of
// each class one SM retires per clock.  The blind rotation is bound by
// integer issue (its NTT butterflies, multiply-accumulates and CRT), so its
// roofline needs these rates measured on the chip rather than assumed.
//
// Every kernel runs, per thread, eight independent dependency chains of one
// operation written as inline PTX (so the compiler can neither fold nor
// reorder them away), long enough that launch overhead is negligible.  One
// thread per CTA records clock64() and %globaltimer at the start and end of
// its CTA's loop, which gives cycles and the SM clock of the run.  The host
// side (bench.py --path peaks) turns lanes x operations / (SMs x cycles)
// into operations per clock per SM.
//
// Separate library (libintpeaks.so): measurement only, not part of the PBS
// path.
#include <cuda_runtime.h>
#include <stdint.h>

namespace {

constexpr int kChains = 8;

__device__ __forceinline__ uint64_t globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// One step of chain x with loop constants a, b: one instruction (two for
// Op<5>).
template <int OP>
struct Op;

template <>
struct Op<0> {  // IADD3: three-input add (two PTX adds fuse into one)
  __device__ __forceinline__ static void step(uint32_t &x, uint32_t a, uint32_t b) {
    asm volatile("{ .reg .u32 t; add.u32 t, %0, %1; add.u32 %0, t, %2; }" : "+r"(x) : "r"(a), "r"(b));
  }
};
template <>
struct Op<1> {  // LOP3: three-input logic (xor of three)
  __device__ __forceinline__ static void step(uint32_t &x, uint32_t a, uint32_t b) {
    asm volatile("lop3.b32 %0, %0, %1, %2, 0x96;" : "+r"(x) : "r"(a), "r"(b));
  }
};
template <>
struct Op<2> {  // IMAD: low 32 bits of x a + b
  __device__ __forceinline__ static void step(uint32_t &x, uint32_t a, uint32_t b) {
    asm volatile("mad.lo.u32 %0, %0, %1, %2;" : "+r"(x) : "r"(a), "r"(b));
  }
};
template <>
struct Op<3> {  // IMAD.HI: high 32 bits of x a, plus b
  __device__ __forceinline__ static void step(uint32_t &x, uint32_t a, uint32_t b) {
    asm volatile("mad.hi.u32 %0, %0, %1, %2;" : "+r"(x) : "r"(a), "r"(b));
  }
};
template <>
struct Op<5> {  // one IMAD and one IADD3 per step (pipe co-issue)
  __device__ __forceinline__ static void step(uint32_t &x, uint32_t a, uint32_t b) {
    asm volatile("{ .reg .u32 t, u; mad.lo.u32 t, %0, %1, %2; add.u32 u, t, %1; add.u32 %0, u, %2; }"
                 : "+r"(x)
                 : "r"(a), "r"(b));
  }
};

template <int OP>
__global__ void __launch_bounds__(512) int_peak_kernel(uint32_t iters, uint32_t seed, uint32_t *sink,
                                                       unsigned long long *stamps) {
  uint32_t x[kChains];
#pragma unroll
  for (int j = 0; j < kChains; ++j) x[j] = seed ^ (threadIdx.x * 2654435761u) ^ (j * 40503u);
  const uint32_t a = seed | 1u, b = seed * 3u + 7u;
  __syncthreads();
  const long long c0 = clock64();
  const uint64_t g0 = globaltimer();
  for (uint32_t i = 0; i < iters; ++i) {
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
      for (int j = 0; j < kChains; ++j) Op<OP>::step(x[j], a, b);
  }
  __syncthreads();
  const long long c1 = clock64();
  const uint64_t g1 = globaltimer();
  uint32_t r = 0;
#pragma unroll
  for (int j = 0; j < kChains; ++j) r ^= x[j];
  if (r == 0x9e3779b9u) sink[0] = r;  // keeps the chains live
  if (threadIdx.x == 0) {
    stamps[2 * blockIdx.x] = static_cast<unsigned long long>(c1 - c0);
    stamps[2 * blockIdx.x + 1] = g1 - g0;
  }
}

// The forward NTT butterfly of the blind rotation (Shoup product, lazy
// range): q = hi(Y ws); t = Y w - q p; Y' = X - t + 2p; X' = X + t.  Eight
// independent butterflies per thread; counted as 5 integer operations (three
// multiplies, two adds).
__global__ void __launch_bounds__(512) bfly_peak_kernel(uint32_t iters, uint32_t seed, uint32_t *sink,
                                                        unsigned long long *stamps) {
  uint32_t X[kChains], Y[kChains];
#pragma unroll
  for (int j = 0; j < kChains; ++j) {
    X[j] = (seed ^ (threadIdx.x * 2654435761u) ^ j) & 0x0FFFFFFFu;
    Y[j] = (seed * 7u + threadIdx.x + j * 977u) & 0x0FFFFFFFu;
  }
  const uint32_t p = 268369921u, w = (seed % p) | 1u;
  const uint32_t ws = static_cast<uint32_t>((static_cast<uint64_t>(w) << 32) / p), two_p = 2 * p;
  __syncthreads();
  const long long c0 = clock64();
  const uint64_t g0 = globaltimer();
  for (uint32_t i = 0; i < iters; ++i) {
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
      for (int j = 0; j < kChains; ++j) {
        uint32_t q, t;
        asm volatile("mul.hi.u32 %0, %1, %2;" : "=r"(q) : "r"(Y[j]), "r"(ws));
        asm volatile("{ .reg .u32 m; mul.lo.u32 m, %1, %2; mad.lo.u32 %0, %3, %4, m; }"
                     : "=r"(t)
                     : "r"(Y[j]), "r"(w), "r"(q), "r"(0u - p));
        const uint32_t yn = X[j] - t + two_p;  // words wrap mod 2^32: the Shoup product
        X[j] = X[j] + t;                       // is valid for any 32-bit Y
        Y[j] = yn;
      }
  }
  __syncthreads();
  const long long c1 = clock64();
  const uint64_t g1 = globaltimer();
  uint32_t r = 0;
#pragma unroll
  for (int j = 0; j < kChains; ++j) r ^= X[j] ^ Y[j];
  if (r == 0x9e3779b9u) sink[0] = r;
  if (threadIdx.x == 0) {
    stamps[2 * blockIdx.x] = static_cast<unsigned long long>(c1 - c0);
    stamps[2 * blockIdx.x + 1] = g1 - g0;
  }
}

// The butterfly three primes near 2^31 would need (products of three such
// primes reach the 92-93 bits the larger parameter sets ask for): 4p no
// longer fits 32 bits, so t and X are brought below p in every butterfly
// before the adds: t = min(t, t - p), X = min(X, X - p), X' = X + t,
// Y' = X - t + p, with the same Shoup product.  Counted as 9 integer
// operations (three multiplies, six adds and minima).
__global__ void __launch_bounds__(512) bfly31_peak_kernel(uint32_t iters, uint32_t seed, uint32_t *sink,
                                                          unsigned long long *stamps) {
  const uint32_t p = 2147352577u;  // 2^31 - 2^17 + 1
  uint32_t X[kChains], Y[kChains];
#pragma unroll
  for (int j = 0; j < kChains; ++j) {
    X[j] = (seed ^ (threadIdx.x * 2654435761u) ^ j) % (2 * p);
    Y[j] = (seed * 7u + threadIdx.x + j * 977u) % (2 * p);
  }
  const uint32_t w = (seed % p) | 1u;
  const uint32_t ws = static_cast<uint32_t>((static_cast<uint64_t>(w) << 32) / p);
  __syncthreads();
  const long long c0 = clock64();
  const uint64_t g0 = globaltimer();
  for (uint32_t i = 0; i < iters; ++i) {
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
      for (int j = 0; j < kChains; ++j) {
        uint32_t q, t;
        asm volatile("mul.hi.u32 %0, %1, %2;" : "=r"(q) : "r"(Y[j]), "r"(ws));
        asm volatile("{ .reg .u32 m; mul.lo.u32 m, %1, %2; mad.lo.u32 %0, %3, %4, m; }"
                     : "=r"(t)
                     : "r"(Y[j]), "r"(w), "r"(q), "r"(0u - p));
        t = min(t, t - p);
        const uint32_t x = min(X[j], X[j] - p);
        X[j] = x + t;
        Y[j] = x - t + p;
      }
  }
  __syncthreads();
  const long long c1 = clock64();
  const uint64_t g1 = globaltimer();
  uint32_t r = 0;
#pragma unroll
  for (int j = 0; j < kChains; ++j) r ^= X[j] ^ Y[j];
  if (r == 0x9e3779b9u) sink[0] = r;
  if (threadIdx.x == 0) {
    stamps[2 * blockIdx.x] = static_cast<unsigned long long>(c1 - c0);
    stamps[2 * blockIdx.x + 1] = g1 - g0;
  }
}

// IMAD.WIDE: 64-bit chains acc = lo(acc) a + acc, so both halves of every
// 32 x 32 -> 64 product are live.
__global__ void __launch_bounds__(512) wide_peak_kernel(uint32_t iters, uint32_t seed, uint32_t *sink,
                                                        unsigned long long *stamps) {
  uint64_t acc[kChains];
#pragma unroll
  for (int j = 0; j < kChains; ++j) acc[j] = seed ^ (threadIdx.x * 0x9E3779B97F4A7C15ull) ^ j;
  const uint32_t a = seed | 1u;
  __syncthreads();
  const long long c0 = clock64();
  const uint64_t g0 = globaltimer();
  for (uint32_t i = 0; i < iters; ++i) {
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
      for (int j = 0; j < kChains; ++j)
        asm volatile("{ .reg .u32 l; cvt.u32.u64 l, %0; mad.wide.u32 %0, l, %1, %0; }" : "+l"(acc[j]) : "r"(a));
  }
  __syncthreads();
  const long long c1 = clock64();
  const uint64_t g1 = globaltimer();
  uint64_t r = 0;
#pragma unroll
  for (int j = 0; j < kChains; ++j) r ^= acc[j];
  if (r == 0x9e3779b97f4a7c15ull) sink[0] = static_cast<uint32_t>(r);
  if (threadIdx.x == 0) {
    stamps[2 * blockIdx.x] = static_cast<unsigned long long>(c1 - c0);
    stamps[2 * blockIdx.x + 1] = g1 - g0;
  }
}

}  // namespace

// Integer operations one thread executes per loop iteration of kernel `op`
// (0 IADD3, 1 LOP3, 2 IMAD, 3 IMAD.HI, 4 IMAD.WIDE, 5 IMAD+IADD3,
// 6 butterfly: 5 integer operations, 7 the butterfly of primes near 2^31:
// 9 integer operations);
// 0 for an unknown op.
extern "C" uint32_t intpeak_ops_per_iter(int op) {
  switch (op) {
    case 0: case 1: case 2: case 3: case 4: return 4 * kChains;
    case 5: return 4 * kChains * 2;
    case 6: return 4 * kChains * 5;
    case 7: return 4 * kChains * 9;
    default: return 0;
  }
}

// Launch kernel `op` on `ctas` CTAs of `threads` threads (<= 512), `iters`
// loop iterations each, on `stream`.  stamps: device buffer of 2*ctas words
// (cycles, nanoseconds per CTA); sink: one device word.  Returns a
// cudaError_t value (0 = success).
extern "C" int intpeak_launch(int op, uint32_t ctas, uint32_t threads, uint32_t iters, uint32_t *sink,
                              unsigned long long *stamps, void *stream) {
  if (threads == 0 || threads > 512 || ctas == 0 || !sink || !stamps) return cudaErrorInvalidValue;
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const uint32_t seed = 0x2545F491u;
  switch (op) {
    case 0: int_peak_kernel<0><<<ctas, threads, 0, s>>>(iters, seed, sink, stamps); break;
    case 1: int_peak_kernel<1><<<ctas, threads, 0, s>>>(iters, seed, sink, stamps); break;
    case 2: int_peak_kernel<2><<<ctas, threads, 0, s>>>(iters, seed, sink, stamps); break;
    case 3: int_peak_kernel<3><<<ctas, threads, 0, s>>>(iters, seed, sink, stamps); break;
    case 4: wide_peak_kernel<<<ctas, threads, 0, s>>>(iters, seed, sink, stamps); break;
    case 5: int_peak_kernel<5><<<ctas, threads, 0, s>>>(iters, seed, sink, stamps); break;
    case 6: bfly_peak_kernel<<<ctas, threads, 0, s>>>(iters, seed, sink, stamps); break;
    case 7: bfly31_peak_kernel<<<ctas, threads, 0, s>>>(iters, seed, sink, stamps); break;
    default: return cudaErrorInvalidValue;
  }
  return static_cast<int>(cudaGetLastError());
}
