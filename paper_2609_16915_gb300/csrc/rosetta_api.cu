// C ABI of librosetta: context creation, key upload, batched PBS, key
// switch.  Validates every argument before enqueuing work and never falls back
// to the host.  Declarations and their documentation: include/rosetta.h.
#include <cuda_runtime.h>

#include <cstring>
#include <new>
#include <vector>

#include "rosetta.h"
#include "context.h"
#include "internal.h"

using namespace rosetta;


namespace {

int cuda_fail(cudaError_t e) {
  return e == cudaErrorMemoryAllocation ? ROSETTA_ERR_OOM : ROSETTA_ERR_CUDA;
}

bool is_device_ptr(const void *p) {
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

bool overlaps(const void *a, size_t na, const void *b, size_t nb) {
  const char *pa = static_cast<const char *>(a), *pb = static_cast<const char *>(b);
  return pa < pb + nb && pb < pa + na;
}

bool aligned8(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 7u) == 0; }

uint32_t log2_exact(uint32_t x) {
  uint32_t r = 0;
  while ((1u << r) < x) ++r;
  return (1u << r) == x ? r : 0xffffffffu;
}

// Number of bits of the largest possible |integer value| of an external
// product coefficient, (k+1) l N 2^(beta-1) 2^63, rounded up.
double ext_product_bits(const rosetta_params &p) {
  double v = 63.0 + (p.pbs_base_log - 1);
  double f = (double)(p.glwe_dim + 1) * p.pbs_level * p.poly_size;
  int e = 0;
  while ((double)(1ull << e) < f) ++e;
  return v + e;
}

// Does the exact integer value of every external-product coefficient,
// |X| <= (k+1) l N 2^(beta-1) 2^63, stay within 0.45 of the product of the
// three 31-bit primes (the margin the three-prime CRT quotient needs)?
bool fits_three_primes(const rosetta_params &p) {
  using u128 = unsigned __int128;
  u128 M3 = 1;
  for (int q = 0; q < kPrimes31; ++q) M3 *= kPrime31List[q];
  const u128 bound = (static_cast<u128>(p.glwe_dim + 1) * p.pbs_level * p.poly_size) << (p.pbs_base_log - 1 + 63);
  return bound * 20 <= M3 * 9;
}

int check_params(const rosetta_params &p) {
  const uint32_t logN = log2_exact(p.poly_size);
  if (logN < 8 || logN > 13) return ROSETTA_ERR_UNSUPPORTED_PARAMS;
  if (p.glwe_dim != 1) return ROSETTA_ERR_UNSUPPORTED_PARAMS;
  if (p.lwe_dim == 0 || p.lwe_dim > 65535) return ROSETTA_ERR_UNSUPPORTED_PARAMS;
  if (p.pbs_base_log < 1 || p.pbs_base_log > 28 || p.pbs_level < 1 || p.pbs_base_log * p.pbs_level > 64)
    return ROSETTA_ERR_UNSUPPORTED_PARAMS;
  if (p.ks_base_log < 1 || p.ks_base_log > 16 || p.ks_level < 1 || p.ks_base_log * p.ks_level > 64)
    return ROSETTA_ERR_UNSUPPORTED_PARAMS;
  if (p.msg_bits < 1 || p.msg_bits > 62 || (p.poly_size >> p.msg_bits) < 2) return ROSETTA_ERR_UNSUPPORTED_PARAMS;
  // exact CRT: the product of the four primes (> 2^111.99) must exceed twice the bound
  if (ext_product_bits(p) + 1.0 > 111.0) return ROSETTA_ERR_UNSUPPORTED_PARAMS;
  return ROSETTA_OK;
}

// (Re)allocate *buf, stream-ordered, to hold at least `need` words.
int ensure(uint64_t **buf, size_t *cap_words, size_t need, cudaStream_t s) {
  if (*buf && *cap_words >= need) return ROSETTA_OK;
  if (*buf) {
    cudaError_t e = cudaFreeAsync(*buf, s);
    *buf = nullptr;
    *cap_words = 0;
    if (e != cudaSuccess) return cuda_fail(e);
  }
  cudaError_t e = cudaMallocAsync(reinterpret_cast<void **>(buf), need * sizeof(uint64_t), s);
  if (e != cudaSuccess) {
    *buf = nullptr;
    return cuda_fail(e);
  }
  *cap_words = need;
  return ROSETTA_OK;
}

size_t lwe_words(const rosetta_ctx *c) { return c->prm.lwe_dim + 1; }
size_t big_words(const rosetta_ctx *c) { return (size_t)c->prm.glwe_dim * c->prm.poly_size + 1; }
size_t stage_words(const rosetta_ctx *c) { return big_words(c) > lwe_words(c) ? big_words(c) : lwe_words(c); }

// Scratch for the extracted ciphertexts of `batch` inputs.
int ensure_big(rosetta_ctx *c, uint32_t batch, cudaStream_t s) {
  return ensure(&c->d_big, &c->big_words_cap, (size_t)batch * big_words(c), s);
}

// Staging for host-memory inputs and outputs of `batch` ciphertexts.
int ensure_stage(rosetta_ctx *c, uint32_t batch, cudaStream_t s) {
  const size_t need = (size_t)batch * stage_words(c);
  int st = ensure(&c->d_in, &c->in_words_cap, need, s);
  return st == ROSETTA_OK ? ensure(&c->d_out, &c->out_words_cap, need, s) : st;
}

cudaStream_t as_stream(void *s) { return reinterpret_cast<cudaStream_t>(s); }

// Shared front half of the entry points that take ciphertexts in and out:
// validation, host staging of inputs.  in_words/out_words are per ciphertext.
struct Staged {
  const uint64_t *in = nullptr;
  const uint64_t *lut = nullptr;
  uint64_t *out = nullptr;
  bool out_host = false;
};

int stage_io(rosetta_ctx *c, const uint64_t *in, size_t in_words, uint32_t batch, const uint64_t *lut,
             uint64_t *out, size_t out_words, cudaStream_t s, Staged *st) {
  if (!aligned8(in) || !aligned8(out) || (lut && !aligned8(lut))) return ROSETTA_ERR_INVALID_ARG;
  const size_t in_bytes = (size_t)batch * in_words * 8, out_bytes = (size_t)batch * out_words * 8;
  if (overlaps(in, in_bytes, out, out_bytes)) return ROSETTA_ERR_INVALID_ARG;
  if (c->prm.max_batch && batch > c->prm.max_batch) return ROSETTA_ERR_INVALID_ARG;
  const bool in_dev = is_device_ptr(in), out_dev = is_device_ptr(out);
  st->in = in;
  st->out = out;
  st->lut = lut;
  if (!in_dev || !out_dev) {
    int r = ensure_stage(c, batch, s);
    if (r != ROSETTA_OK) return r;
  }
  if (!in_dev) {
    cudaError_t e = cudaMemcpyAsync(c->d_in, in, in_bytes, cudaMemcpyHostToDevice, s);
    if (e != cudaSuccess) return cuda_fail(e);
    st->in = c->d_in;
  }
  if (!out_dev) {
    st->out = c->d_out;
    st->out_host = true;
  }
  if (lut && !is_device_ptr(lut)) {
    cudaError_t e = cudaMemcpyAsync(c->d_lut, lut, sizeof(uint64_t) << c->prm.msg_bits, cudaMemcpyHostToDevice, s);
    if (e != cudaSuccess) return cuda_fail(e);
    st->lut = c->d_lut;
  }
  return ROSETTA_OK;
}

int finish_io(rosetta_ctx *c, uint64_t *out, size_t out_words, uint32_t batch, const Staged &st, cudaStream_t s) {
  (void)c;
  if (!st.out_host) return ROSETTA_OK;
  cudaError_t e = cudaMemcpyAsync(out, st.out, (size_t)batch * out_words * 8, cudaMemcpyDeviceToHost, s);
  if (e != cudaSuccess) return cuda_fail(e);
  e = cudaStreamSynchronize(s);
  return e == cudaSuccess ? ROSETTA_OK : cuda_fail(e);
}

BrArgs br_args(const rosetta_ctx *c, const uint64_t *in, uint32_t batch, const uint64_t *lut, uint64_t *big) {
  BrArgs a{};
  a.lwe_in = in;
  a.lut = lut;
  a.lwe_big_out = big;
  br_key_args(c, &a);
  a.n = c->prm.lwe_dim;
  a.level = c->prm.pbs_level;
  a.base_log = c->prm.pbs_base_log;
  a.msg_bits = c->prm.msg_bits;
  a.batch = batch;
  a.num_luts = 1;
  a.err_flag = c->d_err;
  return a;
}

// Batches from this size on take the tensor-core key switch (when exact for
// the parameters); smaller ones the split-K CUDA-core kernel.
constexpr uint32_t kKsTcMinBatch = 256;

KsArgs ks_args(const rosetta_ctx *c, const uint64_t *big, uint32_t batch, uint64_t *out);

cudaError_t run_keyswitch(rosetta_ctx *c, const uint64_t *big, uint32_t batch, uint64_t *out, cudaStream_t s) {
  const rosetta_params &p = c->prm;
  const uint32_t kN = p.glwe_dim * p.poly_size;
  if (c->ks_limbs && c->d_ks_b && batch >= kKsTcMinBatch) {
    const size_t words16 = ks_tc_a_words16(batch, kN, p.ks_level);
    if (ensure(&c->d_ks_a, &c->ks_a_cap, (words16 + 3) / 4, s) != ROSETTA_OK) return cudaErrorMemoryAllocation;
    KsTcArgs a{};
    a.a_tiles = reinterpret_cast<const uint16_t *>(c->d_ks_a);
    a.b_tiles = c->d_ks_b;
    a.big = big;
    a.out = out;
    a.err_flag = c->d_err;
    a.batch = batch;
    a.kN = kN;
    a.n = p.lwe_dim;
    a.k_steps = kN * p.ks_level / 64;
    a.limbs = c->ks_limbs;
    return launch_keyswitch_tc(a, p.ks_base_log, p.ks_level, s);
  }
  return launch_keyswitch(ks_args(c, big, batch, out), s);
}

KsArgs ks_args(const rosetta_ctx *c, const uint64_t *big, uint32_t batch, uint64_t *out) {
  KsArgs k{};
  k.big = big;
  k.out = out;
  k.ksk = c->d_ksk;
  k.corr = c->d_corr;
  k.batch = batch;
  k.kN = c->prm.glwe_dim * c->prm.poly_size;
  k.n = c->prm.lwe_dim;
  k.base_log = c->prm.ks_base_log;
  k.level = c->prm.ks_level;
  return k;
}

// Plaintext products use an exact 64-bit gadget (16 bits x 4 levels) against
// noiseless rows: row comp*4 + l of component comp holds P 2^(64 - (l+1) 16),
// the other component 0 (raw layout [8][2][N]).
constexpr uint32_t kPmBase = 16, kPmLev = 4, kPmRows = 2 * kPmLev;

void pm_rows(uint64_t *raw, const int64_t *P, size_t N) {
  for (size_t w = 0; w < kPmRows * 2 * N; ++w) raw[w] = 0;
  for (uint32_t comp = 0; comp < 2; ++comp)
    for (uint32_t l = 0; l < kPmLev; ++l)
      for (size_t t = 0; t < N; ++t)
        raw[((comp * kPmLev + l) * 2 + comp) * N + t] = static_cast<uint64_t>(P[t]) << (64 - (l + 1) * kPmBase);
}

// out[b] = (P * in_A, P * in_B + add) with P given by its transformed gadget rows.
cudaError_t launch_pm(const rosetta_ctx *c, const uint32_t *key, const uint64_t *add, const uint64_t *in,
                      uint32_t batch, uint64_t *out, cudaStream_t s) {
  TraceArgs a{};
  a.glwe_in = in;
  a.glwe_out = out;
  a.keys = key;
  a.plain_add = add;
  a.tw = c->d_tw;
  a.base_log = kPmBase;
  a.level = kPmRows;
  a.batch = batch;
  a.cc = c->cc;
  return launch_plaintext_mul(a, c->logN, s);
}

TraceArgs trace_args(const rosetta_ctx *c, const uint64_t *in, uint32_t batch, uint64_t *out) {
  TraceArgs a{};
  a.glwe_in = in;
  a.glwe_out = out;
  a.keys = c->d_trk;
  a.tw = c->d_tw;
  a.base_log = c->trk_base_log;
  a.level = c->trk_level;
  a.batch = batch;
  a.cc = c->cc;
  return a;
}

}  // namespace

extern "C" {

const char *rosetta_status_string(int status) {
  switch (status) {
    case ROSETTA_OK: return "ok";
    case ROSETTA_ERR_INVALID_ARG: return "invalid argument";
    case ROSETTA_ERR_UNSUPPORTED_PARAMS: return "unsupported parameters";
    case ROSETTA_ERR_KEYS_MISSING: return "keys not uploaded";
    case ROSETTA_ERR_CUDA: return "CUDA error";
    case ROSETTA_ERR_OOM: return "out of device memory";
    case ROSETTA_ERR_TIMEOUT: return "device wait timed out";
    case ROSETTA_ERR_BOUNDS: return "device-side bounds check failed (debug build)";
    default: return "unknown status";
  }
}

int rosetta_params_init(rosetta_ctx **out, const rosetta_params *p, int cuda_device) {
  if (!out) return ROSETTA_ERR_INVALID_ARG;
  *out = nullptr;
  if (!p) return ROSETTA_ERR_INVALID_ARG;
  int st = check_params(*p);
  if (st != ROSETTA_OK) return st;
  int ndev = 0;
  if (cudaGetDeviceCount(&ndev) != cudaSuccess || cuda_device < 0 || cuda_device >= ndev) {
    cudaGetLastError();
    return ROSETTA_ERR_CUDA;
  }
  if (cudaSetDevice(cuda_device) != cudaSuccess) return ROSETTA_ERR_CUDA;
  const uint32_t logN = log2_exact(p->poly_size);
  const bool dig16 = p->pbs_base_log <= 16;
  int max_smem = 0;
  cudaDeviceGetAttribute(&max_smem, cudaDevAttrMaxSharedMemoryPerBlockOptin, cuda_device);
  if (br_smem_bytes(logN, p->pbs_level, p->lwe_dim, dig16) > (size_t)max_smem) return ROSETTA_ERR_UNSUPPORTED_PARAMS;

  rosetta_ctx *c = new (std::nothrow) rosetta_ctx();
  if (!c) return ROSETTA_ERR_OOM;
  c->prm = *p;
  c->device = cuda_device;
  c->logN = logN;
  c->dig16 = dig16;
  std::vector<uint2> tw((size_t)kPrimes << logN);
  if (!build_tables(logN, kPrimes, tw.data(), &c->cc)) {
    delete c;
    return ROSETTA_ERR_UNSUPPORTED_PARAMS;
  }
  // The blind rotation runs over three 31-bit primes where the bound allows
  // it, the kernel exists for the ring size and level, and as many of its
  // CTAs fit an SM's shared memory as of the four-prime kernel's; over the
  // four 28-bit primes otherwise.
  int smem_sm = 0, smem_rsv = 0;
  cudaDeviceGetAttribute(&smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, cuda_device);
  cudaDeviceGetAttribute(&smem_rsv, cudaDevAttrReservedSharedMemoryPerBlock, cuda_device);
  const size_t smem3 = br3_smem_bytes(logN, p->pbs_level, p->lwe_dim);
  const size_t smem4 = br_smem_bytes(logN, p->pbs_level, p->lwe_dim, dig16);
  const auto per_sm = [&](size_t b) { return (size_t)smem_sm / (b + (size_t)smem_rsv); };
  std::vector<uint2> tw31;
  if (fits_three_primes(*p) && br3_supported(logN, p->pbs_level, dig16) && smem3 <= (size_t)max_smem &&
      per_sm(smem3) >= per_sm(smem4)) {
    tw31.resize((size_t)kPrimes31 << logN);
    if (build_tables(logN, kPrimes31, tw31.data(), &c->cc31)) c->br_primes = kPrimes31;
  }
  cudaError_t e = cudaMalloc(&c->d_tw, tw.size() * sizeof(uint2));
  if (e == cudaSuccess) e = cudaMemcpy(c->d_tw, tw.data(), tw.size() * sizeof(uint2), cudaMemcpyHostToDevice);
  if (e == cudaSuccess && c->br_primes == kPrimes31) {
    e = cudaMalloc(&c->d_tw31, tw31.size() * sizeof(uint2));
    if (e == cudaSuccess)
      e = cudaMemcpy(c->d_tw31, tw31.data(), tw31.size() * sizeof(uint2), cudaMemcpyHostToDevice);
  }
  if (e == cudaSuccess) e = cudaMalloc(&c->d_lut, sizeof(uint64_t) << p->msg_bits);
  if (e == cudaSuccess) e = cudaMalloc(&c->d_err, sizeof(uint32_t));
  if (e == cudaSuccess) e = cudaMemset(c->d_err, 0, sizeof(uint32_t));
  if (e != cudaSuccess) {
    rosetta_destroy(c);
    return cuda_fail(e);
  }
  if (p->max_batch) {
    st = ensure_big(c, p->max_batch, nullptr);
    if (st == ROSETTA_OK) st = ensure_stage(c, p->max_batch, nullptr);
    if (st == ROSETTA_OK && cudaStreamSynchronize(nullptr) != cudaSuccess) st = ROSETTA_ERR_CUDA;
    if (st != ROSETTA_OK) {
      rosetta_destroy(c);
      return st;
    }
  }
  *out = c;
  return ROSETTA_OK;
}

int rosetta_upload_bsk(rosetta_ctx *c, const uint64_t *bsk, size_t n_words, int src_is_device, void *stream) {
  if (!c || !bsk) return ROSETTA_ERR_INVALID_ARG;
  const rosetta_params &p = c->prm;
  const size_t want = (size_t)p.lwe_dim * (p.glwe_dim + 1) * p.pbs_level * (p.glwe_dim + 1) * p.poly_size;
  if (n_words != want || !aligned8(bsk)) return ROSETTA_ERR_INVALID_ARG;
  if (cudaSetDevice(c->device) != cudaSuccess) return ROSETTA_ERR_CUDA;
  cudaStream_t s = as_stream(stream);
  const uint64_t *src = bsk;
  uint64_t *tmp = nullptr;
  cudaError_t e = cudaSuccess;
  if (!src_is_device) {
    e = cudaMallocAsync(reinterpret_cast<void **>(&tmp), want * 8, s);
    if (e != cudaSuccess) return cuda_fail(e);
    e = cudaMemcpyAsync(tmp, bsk, want * 8, cudaMemcpyHostToDevice, s);
    if (e != cudaSuccess) {
      cudaFreeAsync(tmp, s);
      return cuda_fail(e);
    }
    src = tmp;
  }
  // one 32-bit residue per prime of the blind rotation's set for every raw word
  const bool three = c->br_primes == kPrimes31;
  if (!c->d_bsk) e = cudaMalloc(&c->d_bsk, want * c->br_primes * sizeof(uint32_t));
  if (e != cudaSuccess) {
    if (tmp) cudaFreeAsync(tmp, s);
    return cuda_fail(e);
  }
  e = launch_bsk_transform(src, c->d_bsk, three ? c->d_tw31 : c->d_tw, three ? c->cc31 : c->cc, c->logN, p.lwe_dim,
                           p.pbs_level, c->br_primes, s);
  if (tmp) cudaFreeAsync(tmp, s);
  if (e != cudaSuccess) return cuda_fail(e);
  if (!src_is_device) {
    e = cudaStreamSynchronize(s);  // caller may free the host buffer on return
    if (e != cudaSuccess) return cuda_fail(e);
  }
  c->bsk_words = want * c->br_primes;
  c->have_bsk = true;
  return ROSETTA_OK;
}

int rosetta_upload_ksk(rosetta_ctx *c, const uint64_t *ksk, size_t n_words, int src_is_device, void *stream) {
  if (!c || !ksk) return ROSETTA_ERR_INVALID_ARG;
  const rosetta_params &p = c->prm;
  const size_t rows = (size_t)p.glwe_dim * p.poly_size * p.ks_level;
  const size_t want = rows * (p.lwe_dim + 1);
  if (n_words != want || !aligned8(ksk)) return ROSETTA_ERR_INVALID_ARG;
  if (cudaSetDevice(c->device) != cudaSuccess) return ROSETTA_ERR_CUDA;
  cudaStream_t s = as_stream(stream);
  cudaError_t e = cudaSuccess;
  if (!c->d_ksk) e = cudaMalloc(&c->d_ksk, want * 8);
  if (e == cudaSuccess && !c->d_corr) e = cudaMalloc(&c->d_corr, (p.lwe_dim + 1) * 8);
  if (e != cudaSuccess) return cuda_fail(e);
  e = cudaMemcpyAsync(c->d_ksk, ksk, want * 8, src_is_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice, s);
  if (e != cudaSuccess) return cuda_fail(e);
  e = launch_ksk_corr(c->d_ksk, c->d_corr, (uint32_t)rows, p.lwe_dim, p.ks_base_log, s);
  if (e != cudaSuccess) return cuda_fail(e);
  // limb tiles for the tensor-core key switch, where its fp32 sums are exact
  const uint32_t kN = p.glwe_dim * p.poly_size;
  c->ks_limbs = ks_tc_limbs(kN, p.ks_level, p.ks_base_log);
  if (c->ks_limbs) {
    if (!c->d_ks_b) e = cudaMalloc(&c->d_ks_b, ks_tc_b_words16(kN, p.ks_level, p.lwe_dim, c->ks_limbs) * 2);
    if (e == cudaSuccess) e = launch_ks_limbs(c->d_ksk, c->d_ks_b, kN, p.ks_level, p.lwe_dim, c->ks_limbs, s);
    if (e != cudaSuccess) return cuda_fail(e);
  }
  if (!src_is_device) {
    e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e);
  }
  c->have_ksk = true;
  return ROSETTA_OK;
}

int rosetta_blind_rotate_extract_batch(rosetta_ctx *c, const uint64_t *lwe_in, uint32_t batch, const uint64_t *lut,
                                       uint64_t *lwe_big_out, void *stream) {
  if (!c) return ROSETTA_ERR_INVALID_ARG;
  if (batch == 0) return ROSETTA_OK;
  if (!lwe_in || !lut || !lwe_big_out) return ROSETTA_ERR_INVALID_ARG;
  if (!c->have_bsk) return ROSETTA_ERR_KEYS_MISSING;
  if (cudaSetDevice(c->device) != cudaSuccess) return ROSETTA_ERR_CUDA;
  cudaStream_t s = as_stream(stream);
  Staged st;
  int r = stage_io(c, lwe_in, lwe_words(c), batch, lut, lwe_big_out, big_words(c), s, &st);
  if (r != ROSETTA_OK) return r;
  cudaError_t e = launch_blind_rotate(br_args(c, st.in, batch, st.lut, st.out), c->logN, c->dig16, s);
  if (e != cudaSuccess) return cuda_fail(e);
  return finish_io(c, lwe_big_out, big_words(c), batch, st, s);
}

int rosetta_keyswitch_batch(rosetta_ctx *c, const uint64_t *lwe_big_in, uint32_t batch, uint64_t *lwe_out,
                            void *stream) {
  if (!c) return ROSETTA_ERR_INVALID_ARG;
  if (batch == 0) return ROSETTA_OK;
  if (!lwe_big_in || !lwe_out) return ROSETTA_ERR_INVALID_ARG;
  if (!c->have_ksk) return ROSETTA_ERR_KEYS_MISSING;
  if (cudaSetDevice(c->device) != cudaSuccess) return ROSETTA_ERR_CUDA;
  cudaStream_t s = as_stream(stream);
  Staged st;
  int r = stage_io(c, lwe_big_in, big_words(c), batch, nullptr, lwe_out, lwe_words(c), s, &st);
  if (r != ROSETTA_OK) return r;
  cudaError_t e = run_keyswitch(c, st.in, batch, st.out, s);
  if (e != cudaSuccess) return cuda_fail(e);
  return finish_io(c, lwe_out, lwe_words(c), batch, st, s);
}

int rosetta_pbs_batch(rosetta_ctx *c, const uint64_t *lwe_in, uint32_t batch, const uint64_t *lut,
                      uint64_t *lwe_out, void *stream) {
  if (!c) return ROSETTA_ERR_INVALID_ARG;
  if (batch == 0) return ROSETTA_OK;
  if (!lwe_in || !lut || !lwe_out) return ROSETTA_ERR_INVALID_ARG;
  if (!c->have_bsk || !c->have_ksk) return ROSETTA_ERR_KEYS_MISSING;
  if (cudaSetDevice(c->device) != cudaSuccess) return ROSETTA_ERR_CUDA;
  cudaStream_t s = as_stream(stream);
  Staged st;
  int r = stage_io(c, lwe_in, lwe_words(c), batch, lut, lwe_out, lwe_words(c), s, &st);
  if (r != ROSETTA_OK) return r;
  r = ensure_big(c, batch, s);
  if (r != ROSETTA_OK) return r;
  cudaError_t e = launch_blind_rotate(br_args(c, st.in, batch, st.lut, c->d_big), c->logN, c->dig16, s);
  if (e != cudaSuccess) return cuda_fail(e);
  e = run_keyswitch(c, c->d_big, batch, st.out, s);
  if (e != cudaSuccess) return cuda_fail(e);
  return finish_io(c, lwe_out, lwe_words(c), batch, st, s);
}

int rosetta_pbs_batch_multi_lut(rosetta_ctx *c, const uint64_t *lwe_in, uint32_t batch, const uint64_t *luts,
                                uint32_t num_luts, const uint32_t *lut_index, uint64_t *lwe_out, void *stream) {
  if (!c) return ROSETTA_ERR_INVALID_ARG;
  if (batch == 0) return ROSETTA_OK;
  if (!lwe_in || !luts || !lut_index || !lwe_out || num_luts == 0) return ROSETTA_ERR_INVALID_ARG;
  if (!c->have_bsk || !c->have_ksk) return ROSETTA_ERR_KEYS_MISSING;
  if (cudaSetDevice(c->device) != cudaSuccess) return ROSETTA_ERR_CUDA;
  // the LUT table and the index array are read by the kernel directly
  if (!is_device_ptr(luts) || !is_device_ptr(lut_index) || !aligned8(luts) ||
      (reinterpret_cast<uintptr_t>(lut_index) & 3u))
    return ROSETTA_ERR_INVALID_ARG;
  cudaStream_t s = as_stream(stream);
  Staged st;
  int r = stage_io(c, lwe_in, lwe_words(c), batch, nullptr, lwe_out, lwe_words(c), s, &st);
  if (r != ROSETTA_OK) return r;
  r = ensure_big(c, batch, s);
  if (r != ROSETTA_OK) return r;
  BrArgs a = br_args(c, st.in, batch, luts, c->d_big);
  a.lut_index = lut_index;
  a.num_luts = num_luts;
  cudaError_t e = launch_blind_rotate(a, c->logN, c->dig16, s);
  if (e != cudaSuccess) return cuda_fail(e);
  e = run_keyswitch(c, c->d_big, batch, st.out, s);
  if (e != cudaSuccess) return cuda_fail(e);
  return finish_io(c, lwe_out, lwe_words(c), batch, st, s);
}

int rosetta_blind_rotate_glwe_batch(rosetta_ctx *c, const uint64_t *lwe_in, uint32_t batch, const uint64_t *glwe_in,
                                    uint64_t *glwe_out, void *stream) {
  if (!c) return ROSETTA_ERR_INVALID_ARG;
  if (batch == 0) return ROSETTA_OK;
  if (!lwe_in || !glwe_in || !glwe_out) return ROSETTA_ERR_INVALID_ARG;
  if (!c->have_bsk) return ROSETTA_ERR_KEYS_MISSING;
  if (cudaSetDevice(c->device) != cudaSuccess) return ROSETTA_ERR_CUDA;
  const size_t gw = 2 * (size_t)c->prm.poly_size;
  if (!is_device_ptr(lwe_in) || !is_device_ptr(glwe_in) || !is_device_ptr(glwe_out) || !aligned8(lwe_in) ||
      !aligned8(glwe_in) || !aligned8(glwe_out))
    return ROSETTA_ERR_INVALID_ARG;
  const size_t gbytes = (size_t)batch * gw * 8;
  if (overlaps(glwe_in, gbytes, glwe_out, gbytes) || overlaps(lwe_in, (size_t)batch * lwe_words(c) * 8, glwe_out, gbytes))
    return ROSETTA_ERR_INVALID_ARG;
  BrArgs a = br_args(c, lwe_in, batch, nullptr, nullptr);
  a.glwe_in = glwe_in;
  a.glwe_out = glwe_out;
  cudaError_t e = launch_blind_rotate(a, c->logN, c->dig16, as_stream(stream));
  return e == cudaSuccess ? ROSETTA_OK : cuda_fail(e);
}

int rosetta_upload_trace_keys(rosetta_ctx *c, const uint64_t *keys, size_t n_words, uint32_t base_log,
                              uint32_t level, int src_is_device, void *stream) {
  if (!c || !keys) return ROSETTA_ERR_INVALID_ARG;
  const rosetta_params &p = c->prm;
  if (base_log < 1 || base_log > 28 || level < 2 || (level & 1u) || base_log * level > 64)
    return ROSETTA_ERR_UNSUPPORTED_PARAMS;
  if (c->logN > 12) return ROSETTA_ERR_UNSUPPORTED_PARAMS;
  // exact CRT: level N 2^(base_log-1) 2^63 below M/2 > 2^114
  {
    int e = 0;
    while ((1ull << e) < (uint64_t)level * p.poly_size) ++e;
    if (63 + (base_log - 1) + e + 1 > 111) return ROSETTA_ERR_UNSUPPORTED_PARAMS;
  }
  int max_smem = 0;
  cudaDeviceGetAttribute(&max_smem, cudaDevAttrMaxSharedMemoryPerBlockOptin, c->device);
  if (trace_smem_bytes(c->logN, level) > (size_t)max_smem) return ROSETTA_ERR_UNSUPPORTED_PARAMS;
  const size_t want = (size_t)c->logN * level * 2 * p.poly_size;
  if (n_words != want || !aligned8(keys)) return ROSETTA_ERR_INVALID_ARG;
  if (cudaSetDevice(c->device) != cudaSuccess) return ROSETTA_ERR_CUDA;
  cudaStream_t s = as_stream(stream);
  const uint64_t *src = keys;
  uint64_t *tmp = nullptr;
  cudaError_t e = cudaSuccess;
  if (!src_is_device) {
    e = cudaMallocAsync(reinterpret_cast<void **>(&tmp), want * 8, s);
    if (e != cudaSuccess) return cuda_fail(e);
    e = cudaMemcpyAsync(tmp, keys, want * 8, cudaMemcpyHostToDevice, s);
    if (e != cudaSuccess) {
      cudaFreeAsync(tmp, s);
      return cuda_fail(e);
    }
    src = tmp;
  }
  if (c->d_trk && c->trk_level != level) {
    cudaFree(c->d_trk);
    c->d_trk = nullptr;
  }
  if (!c->d_trk) e = cudaMalloc(&c->d_trk, want * kPrimes * sizeof(uint32_t));
  if (e != cudaSuccess) {
    if (tmp) cudaFreeAsync(tmp, s);
    return cuda_fail(e);
  }
  e = launch_key_transform(src, c->d_trk, c->d_tw, c->cc, c->logN, c->logN, level, s);
  if (tmp) cudaFreeAsync(tmp, s);
  if (e != cudaSuccess) return cuda_fail(e);
  if (!src_is_device) {
    e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e);
  }
  c->trk_base_log = base_log;
  c->trk_level = level;
  c->have_trk = true;
  return ROSETTA_OK;
}

int rosetta_trace_batch(rosetta_ctx *c, const uint64_t *glwe_in, uint32_t batch, uint64_t *glwe_out, void *stream) {
  if (!c) return ROSETTA_ERR_INVALID_ARG;
  if (batch == 0) return ROSETTA_OK;
  if (!glwe_in || !glwe_out) return ROSETTA_ERR_INVALID_ARG;
  if (!c->have_trk) return ROSETTA_ERR_KEYS_MISSING;
  if (cudaSetDevice(c->device) != cudaSuccess) return ROSETTA_ERR_CUDA;
  const size_t gbytes = (size_t)batch * 2 * c->prm.poly_size * 8;
  if (!is_device_ptr(glwe_in) || !is_device_ptr(glwe_out) || !aligned8(glwe_in) || !aligned8(glwe_out) ||
      overlaps(glwe_in, gbytes, glwe_out, gbytes))
    return ROSETTA_ERR_INVALID_ARG;
  cudaError_t e = launch_trace(trace_args(c, glwe_in, batch, glwe_out), c->logN, as_stream(stream));
  return e == cudaSuccess ? ROSETTA_OK : cuda_fail(e);
}

int rosetta_plaintext_mul_batch(rosetta_ctx *c, const uint64_t *glwe_in, uint32_t batch, const int64_t *plain_mul,
                                const uint64_t *plain_add, uint64_t *glwe_out, void *stream) {
  if (!c) return ROSETTA_ERR_INVALID_ARG;
  if (batch == 0) return ROSETTA_OK;
  if (!glwe_in || !plain_mul || !glwe_out) return ROSETTA_ERR_INVALID_ARG;
  if (c->logN > 12 || c->prm.glwe_dim != 1) return ROSETTA_ERR_UNSUPPORTED_PARAMS;
  if (cudaSetDevice(c->device) != cudaSuccess) return ROSETTA_ERR_CUDA;
  const size_t N = c->prm.poly_size;
  const size_t gbytes = (size_t)batch * 2 * N * 8;
  if (!is_device_ptr(glwe_in) || !is_device_ptr(glwe_out) || !aligned8(glwe_in) || !aligned8(glwe_out) ||
      !aligned8(plain_mul) || (plain_add && !aligned8(plain_add)) || overlaps(glwe_in, gbytes, glwe_out, gbytes))
    return ROSETTA_ERR_INVALID_ARG;
  if (is_device_ptr(plain_mul)) return ROSETTA_ERR_INVALID_ARG;  // the gadget rows are built on the host
  std::vector<uint64_t> raw(kPmRows * 2 * N);
  pm_rows(raw.data(), plain_mul, N);
  cudaStream_t s = as_stream(stream);
  cudaError_t e = cudaSuccess;
  if (!c->d_pm_raw) e = cudaMalloc(&c->d_pm_raw, raw.size() * 8);
  if (e == cudaSuccess && !c->d_pm_key) e = cudaMalloc(&c->d_pm_key, raw.size() * kPrimes * sizeof(uint32_t));
  if (e == cudaSuccess && !c->d_pm_add) e = cudaMalloc(&c->d_pm_add, N * 8);
  if (e != cudaSuccess) return cuda_fail(e);
  e = cudaMemcpyAsync(c->d_pm_raw, raw.data(), raw.size() * 8, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess && plain_add)
    e = cudaMemcpyAsync(c->d_pm_add, plain_add, N * 8, cudaMemcpyDefault, s);
  if (e == cudaSuccess) e = launch_key_transform(c->d_pm_raw, c->d_pm_key, c->d_tw, c->cc, c->logN, 1, kPmRows, s);
  if (e == cudaSuccess) e = launch_pm(c, c->d_pm_key, plain_add ? c->d_pm_add : nullptr, glwe_in, batch, glwe_out, s);
  if (e != cudaSuccess) return cuda_fail(e);
  e = cudaStreamSynchronize(s);  // the host staging vector goes out of scope
  return e == cudaSuccess ? ROSETTA_OK : cuda_fail(e);
}

int rosetta_upload_lookup_table(rosetta_ctx *c, uint32_t n_seg, const int64_t *p_hat, const uint64_t *q_hat,
                                const int64_t *a_hat, const uint64_t *b_hat, void *stream) {
  if (!c || !p_hat || !q_hat || !a_hat || !b_hat) return ROSETTA_ERR_INVALID_ARG;
  const size_t N = c->prm.poly_size;
  if (c->logN > 12 || c->prm.glwe_dim != 1) return ROSETTA_ERR_UNSUPPORTED_PARAMS;
  if (n_seg == 0 || n_seg > 256 || (n_seg & (n_seg - 1)) || n_seg > N) return ROSETTA_ERR_UNSUPPORTED_PARAMS;
  if (is_device_ptr(p_hat) || is_device_ptr(q_hat) || is_device_ptr(a_hat) || is_device_ptr(b_hat))
    return ROSETTA_ERR_INVALID_ARG;  // the tables are encoded on the host
  if (cudaSetDevice(c->device) != cudaSuccess) return ROSETTA_ERR_CUDA;
  const uint32_t polys = n_seg + 2;  // P, A_0 .. A_{n_seg-1}, Box_0
  const size_t poly_words = kPmRows * 2 * N;
  std::vector<uint64_t> raw(polys * poly_words);
  pm_rows(raw.data(), p_hat, N);
  for (uint32_t sg = 0; sg < n_seg; ++sg) pm_rows(raw.data() + (1 + sg) * poly_words, a_hat + sg * N, N);
  // Box_0: the coefficients a rotation by less than half a segment box brings to
  // position 0 (+1 on [0, h), -1 on [N - h, N) by X^N = -1), h = N / (2 n_seg)
  std::vector<int64_t> box(N, 0);
  const size_t h = N / n_seg / 2;
  box[0] = 1;
  for (size_t t = 1; t < h; ++t) box[t] = 1;
  for (size_t t = N - h; t < N; ++t) box[t] = -1;
  pm_rows(raw.data() + (1 + n_seg) * poly_words, box.data(), N);
  std::vector<uint64_t> add((1 + n_seg) * N);
  for (size_t t = 0; t < N; ++t) add[t] = q_hat[t];
  for (size_t w = 0; w < n_seg * N; ++w) add[N + w] = b_hat[w];

  cudaStream_t s = as_stream(stream);
  cudaError_t e = cudaStreamSynchronize(s);  // no lookup in flight reads the old tables
  uint64_t *d_raw = nullptr;
  if (e == cudaSuccess) e = cudaMalloc(&d_raw, raw.size() * 8);
  if (e != cudaSuccess) return cuda_fail(e);
  cudaFree(c->d_lk_key);
  cudaFree(c->d_lk_add);
  c->d_lk_key = nullptr;
  c->d_lk_add = nullptr;
  c->have_lk = false;
  e = cudaMalloc(&c->d_lk_key, raw.size() * kPrimes * sizeof(uint32_t));
  if (e == cudaSuccess) e = cudaMalloc(&c->d_lk_add, add.size() * 8);
  if (e == cudaSuccess) e = cudaMemcpyAsync(d_raw, raw.data(), raw.size() * 8, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) e = cudaMemcpyAsync(c->d_lk_add, add.data(), add.size() * 8, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) e = launch_key_transform(d_raw, c->d_lk_key, c->d_tw, c->cc, c->logN, polys, kPmRows, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  cudaFree(d_raw);
  if (e != cudaSuccess) return cuda_fail(e);
  c->lk_nseg = n_seg;
  c->have_lk = true;
  return ROSETTA_OK;
}

int rosetta_segmented_lookup_batch(rosetta_ctx *c, const uint64_t *glwe_x, const uint64_t *lwe_seg, uint32_t batch,
                                   uint64_t *glwe_out, void *stream) {
  if (!c) return ROSETTA_ERR_INVALID_ARG;
  if (batch == 0) return ROSETTA_OK;
  if (!glwe_x || !lwe_seg || !glwe_out) return ROSETTA_ERR_INVALID_ARG;
  if (!c->have_bsk || !c->have_ksk || !c->have_trk || !c->have_lk) return ROSETTA_ERR_KEYS_MISSING;
  if (cudaSetDevice(c->device) != cudaSuccess) return ROSETTA_ERR_CUDA;
  const size_t N = c->prm.poly_size, gw = 2 * N;
  const size_t gbytes = (size_t)batch * gw * 8, lbytes = (size_t)batch * lwe_words(c) * 8;
  if (!is_device_ptr(glwe_x) || !is_device_ptr(lwe_seg) || !is_device_ptr(glwe_out) || !aligned8(glwe_x) ||
      !aligned8(lwe_seg) || !aligned8(glwe_out) || overlaps(glwe_x, gbytes, glwe_out, gbytes) ||
      overlaps(lwe_seg, lbytes, glwe_out, gbytes))
    return ROSETTA_ERR_INVALID_ARG;
  cudaStream_t s = as_stream(stream);
  int r = ensure(&c->d_lk_t, &c->lk_t_cap, batch * gw, s);
  if (r == ROSETTA_OK) r = ensure(&c->d_lk_u, &c->lk_u_cap, batch * gw, s);
  if (r == ROSETTA_OK) r = ensure(&c->d_lk_R, &c->lk_R_cap, batch * gw, s);
  if (r == ROSETTA_OK) r = ensure(&c->d_lk_I, &c->lk_I_cap, batch * lwe_words(c), s);
  if (r == ROSETTA_OK) r = ensure_big(c, batch, s);
  if (r != ROSETTA_OK) return r;
  const uint32_t nseg = c->lk_nseg;
  const size_t key_words = (size_t)kPrimes * kPmRows * gw;
  const uint32_t *kP = c->d_lk_key, *kBox = c->d_lk_key + (1 + nseg) * key_words;
  uint64_t *T = c->d_lk_t, *U = c->d_lk_u, *R = c->d_lk_R, *I = c->d_lk_I;

  // Step 2: t = p(X) [[x]] + q(X); PBS of t selected by [[S]] gives [[I]]
  cudaError_t e = launch_pm(c, kP, c->d_lk_add, glwe_x, batch, T, s);
  if (e == cudaSuccess) {
    BrArgs a = br_args(c, lwe_seg, batch, nullptr, c->d_big);
    a.glwe_in = T;
    e = launch_blind_rotate(a, c->logN, c->dig16, s);
  }
  if (e == cudaSuccess) e = run_keyswitch(c, c->d_big, batch, I, s);
  // Step 3, phase 1: r_s = a_s(X) [[x]] + b_s(X), rotated by [[I]], traced, and
  // accumulated as R = sum_s X^(s box) r_s
  const uint32_t seg_box = static_cast<uint32_t>(N / nseg);
  for (uint32_t sg = 0; sg < nseg && e == cudaSuccess; ++sg) {
    e = launch_pm(c, c->d_lk_key + (1 + sg) * key_words, c->d_lk_add + (1 + sg) * N, glwe_x, batch, T, s);
    if (e == cudaSuccess) {
      BrArgs a = br_args(c, I, batch, nullptr, nullptr);
      a.glwe_in = T;
      a.glwe_out = U;
      e = launch_blind_rotate(a, c->logN, c->dig16, s);
    }
    if (e == cudaSuccess) e = launch_trace(trace_args(c, U, batch, T), c->logN, s);
    if (e == cudaSuccess) e = launch_monomial_acc(R, T, 2 * batch, c->logN, sg * seg_box, sg == 0, s);
  }
  // phase 2: spread each value over its segment box, rotate by [[S]], trace
  if (e == cudaSuccess) e = launch_pm(c, kBox, nullptr, R, batch, T, s);
  if (e == cudaSuccess) {
    BrArgs a = br_args(c, lwe_seg, batch, nullptr, nullptr);
    a.glwe_in = T;
    a.glwe_out = U;
    e = launch_blind_rotate(a, c->logN, c->dig16, s);
  }
  if (e == cudaSuccess) e = launch_trace(trace_args(c, U, batch, glwe_out), c->logN, s);
  return e == cudaSuccess ? ROSETTA_OK : cuda_fail(e);
}

int rosetta_ntt_primes(const rosetta_ctx *c) { return c ? static_cast<int>(c->br_primes) : ROSETTA_ERR_INVALID_ARG; }

int rosetta_selftest_wait_timeout(rosetta_ctx *c, uint32_t limit_us, void *stream) {
  if (!c || limit_us == 0 || limit_us > 1000000) return ROSETTA_ERR_INVALID_ARG;
  if (cudaSetDevice(c->device) != cudaSuccess) return ROSETTA_ERR_CUDA;
  cudaError_t e = launch_wait_selftest(c->d_err, limit_us, as_stream(stream));
  return e == cudaSuccess ? ROSETTA_OK : cuda_fail(e);
}

int rosetta_sync_status(rosetta_ctx *c, void *stream) {
  if (!c) return ROSETTA_ERR_INVALID_ARG;
  if (cudaSetDevice(c->device) != cudaSuccess) return ROSETTA_ERR_CUDA;
  cudaError_t e = cudaStreamSynchronize(as_stream(stream));
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e);
  // an out-of-range LUT index seen by a kernel is reported once, then cleared
  uint32_t flag = 0;
  e = cudaMemcpy(&flag, c->d_err, sizeof(flag), cudaMemcpyDeviceToHost);
  if (e == cudaSuccess && flag) e = cudaMemset(c->d_err, 0, sizeof(flag));
  if (e != cudaSuccess) return cuda_fail(e);
  // 1: a LUT index out of range; 2: a bounded device-side wait gave up;
  // 3: a bounds check of a ROSETTA_DEBUG build failed (the access was skipped)
  if (flag == 2) return ROSETTA_ERR_TIMEOUT;
  if (flag == 3) return ROSETTA_ERR_BOUNDS;
  return flag ? ROSETTA_ERR_INVALID_ARG : ROSETTA_OK;
}

int rosetta_selftest_bounds(rosetta_ctx *c, void *stream) {
  if (!c) return ROSETTA_ERR_INVALID_ARG;
#ifndef ROSETTA_DEBUG
  (void)stream;
  return ROSETTA_ERR_UNSUPPORTED_PARAMS;  // the checks exist only in a ROSETTA_DEBUG build
#else
  if (!c->have_bsk) return ROSETTA_ERR_KEYS_MISSING;
  if (cudaSetDevice(c->device) != cudaSuccess) return ROSETTA_ERR_CUDA;
  const cudaStream_t s = as_stream(stream);
  // One ciphertext whose only nonzero mask word is the last (a~ = N, so only
  // the last CMux step runs), blind-rotated with the transformed key declared
  // one step's block shorter than it is: that step's key block fails its
  // check, the kernel skips the loads (it reads nothing past what it is
  // told exists) and raises the flag.
  int r = ensure_stage(c, 1, s);
  if (r == ROSETTA_OK) r = ensure_big(c, 1, s);
  if (r != ROSETTA_OK) return r;
  const uint64_t word = 1ull << 63;
  cudaError_t e = cudaMemsetAsync(c->d_in, 0, lwe_words(c) * sizeof(uint64_t), s);
  if (e == cudaSuccess) e = cudaMemcpyAsync(c->d_in + c->prm.lwe_dim - 1, &word, sizeof(word), cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) e = cudaMemsetAsync(c->d_lut, 0, sizeof(uint64_t) << c->prm.msg_bits, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);  // `word` lives on this stack frame
  if (e != cudaSuccess) return cuda_fail(e);
  BrArgs a = br_args(c, c->d_in, 1, c->d_lut, c->d_big);
  const size_t step = c->bsk_words / c->prm.lwe_dim;
  a.bsk_words = c->bsk_words - step;
  e = launch_blind_rotate(a, c->logN, c->dig16, s);
  return e == cudaSuccess ? ROSETTA_OK : cuda_fail(e);
#endif
}

void rosetta_destroy(rosetta_ctx *c) {
  if (!c) return;
  cudaSetDevice(c->device);
  cudaDeviceSynchronize();
  cudaFree(c->d_tw);
  cudaFree(c->d_tw31);
  cudaFree(c->d_bsk);
  cudaFree(c->d_ksk);
  cudaFree(c->d_corr);
  cudaFree(c->d_ks_b);
  cudaFree(c->d_ks_a);
  cudaFree(c->d_big);
  cudaFree(c->d_in);
  cudaFree(c->d_out);
  cudaFree(c->d_lut);
  cudaFree(c->d_err);
  cudaFree(c->d_trk);
  cudaFree(c->d_pm_raw);
  cudaFree(c->d_pm_key);
  cudaFree(c->d_pm_add);
  cudaFree(c->d_lk_key);
  cudaFree(c->d_lk_add);
  cudaFree(c->d_lk_t);
  cudaFree(c->d_lk_u);
  cudaFree(c->d_lk_R);
  cudaFree(c->d_lk_I);
  delete c;
}

}  // extern "C"
