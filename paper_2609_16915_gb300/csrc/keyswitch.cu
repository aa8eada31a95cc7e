// LWE key switch from dimension kN to n for a batch of ciphertexts:
//   out = (0,..,0,b') - sum_i sum_lev d_{i,lev}(a'_i) * KSK[i][lev]   (mod 2^64)
// with d the signed base-2^beta digits of a'_i rounded to its top beta*l bits.
//
// This is a batched integer matrix product [batch x kN*l] digits times
// [kN*l x (n+1)] key words.  Small batches split the kN input words over
// several CTAs (split-K); the partial sums are combined with 64-bit atomic
// adds, which are exact and order-independent mod 2^64.  Digits are shifted to d + B/2 in [0, B) so every
// product is an unsigned 32x64-bit multiply; the shift is undone with the
// precomputed column sums corr[o] = (B/2) sum_rows KSK[row][o].  Each product
// d * g mod 2^64 is split as d*g_lo (64-bit accumulator) + 2^32 (d*g_hi)
// (a 32-bit accumulator, only its low word matters): two multiply-adds.
#include "internal.h"

namespace rosetta {

namespace {
// 64 ciphertexts x 64 output words per CTA; 128 threads, each 8 ciphertexts x
// 4 consecutive output words; KS_KI input coefficients (KS_KI * l rows of the
// KSK) per shared-memory tile.
constexpr int KS_BM = 64, KS_BN = 64, KS_TM = 8, KS_TN = 4, KS_KI = 8;
constexpr int KS_THREADS = (KS_BM / KS_TM) * (KS_BN / KS_TN);
}  // namespace

__global__ void __launch_bounds__(KS_THREADS) keyswitch_kernel(const KsArgs a) {
  extern __shared__ __align__(16) unsigned char smem[];
  const uint32_t level = a.level;
  uint64_t *ks = reinterpret_cast<uint64_t *>(smem);                          // [KI*level][BN]
  uint32_t *dg = reinterpret_cast<uint32_t *>(ks + KS_KI * level * KS_BN);    // [KI*level][BM]
  const uint32_t tid = threadIdx.x;
  const uint32_t tx = tid % (KS_BN / KS_TN), ty = tid / (KS_BN / KS_TN);
  const uint32_t b0 = blockIdx.y * KS_BM, o0 = blockIdx.x * KS_BN;
  const uint32_t n1 = a.n + 1, stride_in = a.kN + 1;
  const uint32_t bits = a.base_log * level;
  const uint64_t Bmask = (1ull << a.base_log) - 1, Bhalf = 1ull << (a.base_log - 1);

  uint64_t lo[KS_TM][KS_TN];
  uint32_t hi[KS_TM][KS_TN];
#pragma unroll
  for (int m = 0; m < KS_TM; ++m)
#pragma unroll
    for (int t = 0; t < KS_TN; ++t) {
      lo[m][t] = 0;
      hi[m][t] = 0;
    }

  const uint32_t krows = KS_KI * level;
  // this CTA's share of the input words: [i_begin, i_end), KS_KI-aligned
  const uint32_t chunks = (a.kN + KS_KI - 1) / KS_KI;
  const uint32_t per = (chunks + gridDim.z - 1) / gridDim.z;
  const uint32_t i_begin = blockIdx.z * per * KS_KI;
  const uint32_t i_end = min(a.kN, i_begin + per * KS_KI);
  for (uint32_t i0 = i_begin; i0 < i_end; i0 += KS_KI) {
    __syncthreads();
    for (uint32_t idx = tid; idx < KS_BM * KS_KI; idx += KS_THREADS) {
      const uint32_t ii = idx % KS_KI, m = idx / KS_KI;  // consecutive words of one ciphertext
      const uint32_t b = b0 + m, i = i0 + ii;
      const uint64_t v = (b < a.batch && i < a.kN) ? a.big[static_cast<size_t>(b) * stride_in + i] : 0;
      uint64_t cv = bits >= 64 ? v : (v + (1ull << (63 - bits))) >> (64 - bits);
      for (int l = static_cast<int>(level) - 1; l >= 0; --l) {
        const uint64_t d = cv & Bmask;
        cv >>= a.base_log;
        if (d >= Bhalf) cv += 1;
        // the balanced digit d or d - B, shifted by B/2 into [0, B)
        dg[(ii * level + l) * KS_BM + m] = static_cast<uint32_t>((d + Bhalf) & Bmask);
      }
    }
    for (uint32_t idx = tid; idx < krows * KS_BN; idx += KS_THREADS) {
      const uint32_t kr = idx / KS_BN, col = idx % KS_BN;
      const uint32_t i = i0 + kr / level, o = o0 + col;
      ks[idx] = (i < a.kN && o < n1) ? a.ksk[(static_cast<size_t>(i) * level + kr % level) * n1 + o] : 0;
    }
    __syncthreads();
    for (uint32_t kr = 0; kr < krows; ++kr) {
      const uint4 d0 = *reinterpret_cast<const uint4 *>(dg + kr * KS_BM + ty * KS_TM);
      const uint4 d1 = *reinterpret_cast<const uint4 *>(dg + kr * KS_BM + ty * KS_TM + 4);
      const uint4 g01 = *reinterpret_cast<const uint4 *>(ks + kr * KS_BN + tx * KS_TN);
      const uint4 g23 = *reinterpret_cast<const uint4 *>(ks + kr * KS_BN + tx * KS_TN + 2);
      const uint32_t d[KS_TM] = {d0.x, d0.y, d0.z, d0.w, d1.x, d1.y, d1.z, d1.w};
      const uint32_t glo[KS_TN] = {g01.x, g01.z, g23.x, g23.z};
      const uint32_t ghi[KS_TN] = {g01.y, g01.w, g23.y, g23.w};
#pragma unroll
      for (int m = 0; m < KS_TM; ++m)
#pragma unroll
        for (int t = 0; t < KS_TN; ++t) {
          lo[m][t] += static_cast<uint64_t>(d[m]) * glo[t];
          hi[m][t] += d[m] * ghi[t];
        }
    }
  }
#pragma unroll
  for (int m = 0; m < KS_TM; ++m) {
    const uint32_t b = b0 + ty * KS_TM + m;
    if (b >= a.batch) continue;
#pragma unroll
    for (int t = 0; t < KS_TN; ++t) {
      const uint32_t o = o0 + tx * KS_TN + t;
      if (o >= n1) continue;
      const uint64_t sum = lo[m][t] + (static_cast<uint64_t>(hi[m][t]) << 32);
      if (gridDim.z == 1) {
        const uint64_t body = (o == a.n) ? a.big[static_cast<size_t>(b) * stride_in + a.kN] : 0;
        a.out[static_cast<size_t>(b) * n1 + o] = body - sum + a.corr[o];
      } else {
        // the output was zeroed; split 0 also adds the body and the correction
        uint64_t v = 0ull - sum;
        if (blockIdx.z == 0) v += ((o == a.n) ? a.big[static_cast<size_t>(b) * stride_in + a.kN] : 0) + a.corr[o];
        atomicAdd(reinterpret_cast<unsigned long long *>(a.out + static_cast<size_t>(b) * n1 + o),
                  static_cast<unsigned long long>(v));
      }
    }
  }
}

cudaError_t launch_keyswitch(const KsArgs &a, cudaStream_t s) {
  const size_t smem = static_cast<size_t>(KS_KI) * a.level * (KS_BN * sizeof(uint64_t) + KS_BM * sizeof(uint32_t));
  cudaError_t e =
      cudaFuncSetAttribute(keyswitch_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  dim3 grid((a.n + 1 + KS_BN - 1) / KS_BN, (a.batch + KS_BM - 1) / KS_BM, 1);
  // enough CTAs to keep every SM streaming key words: split the input words
  // when the output tiles alone give fewer than ~4 CTAs per SM
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const uint32_t tiles = grid.x * grid.y, want = 4u * static_cast<uint32_t>(sms > 0 ? sms : 1);
  const uint32_t chunks = (a.kN + KS_KI - 1) / KS_KI;
  uint32_t splits = tiles >= want ? 1u : (want + tiles - 1) / tiles;
  if (splits > chunks) splits = chunks;
  splits = (chunks + (chunks + splits - 1) / splits - 1) / ((chunks + splits - 1) / splits);  // no empty splits
  if (splits > 1) {
    grid.z = splits;
    e = cudaMemsetAsync(a.out, 0, static_cast<size_t>(a.batch) * (a.n + 1) * sizeof(uint64_t), s);
    if (e != cudaSuccess) return e;
  }
  keyswitch_kernel<<<grid, KS_THREADS, smem, s>>>(a);
  return cudaGetLastError();
}

// corr[o] = (B/2) * sum_rows ksk[row][o]  (mod 2^64)
__global__ void ksk_corr_kernel(const uint64_t *__restrict__ ksk, uint64_t *__restrict__ corr, uint32_t rows,
                                uint32_t n1, uint64_t half) {
  const uint32_t o = blockIdx.x * blockDim.x + threadIdx.x;
  if (o >= n1) return;
  uint64_t s = 0;
  for (uint32_t r = 0; r < rows; ++r) s += ksk[static_cast<size_t>(r) * n1 + o];
  corr[o] = s * half;
}

cudaError_t launch_ksk_corr(const uint64_t *ksk, uint64_t *corr, uint32_t rows, uint32_t n, uint32_t base_log,
                            cudaStream_t s) {
  const uint32_t n1 = n + 1;
  ksk_corr_kernel<<<(n1 + 127) / 128, 128, 0, s>>>(ksk, corr, rows, n1, 1ull << (base_log - 1));
  return cudaGetLastError();
}

}  // namespace rosetta
