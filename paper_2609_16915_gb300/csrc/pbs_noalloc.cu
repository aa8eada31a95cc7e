// rosetta_pbs_batch_noalloc: batched PBS for callers that must not allocate
// device memory during the call.
//
// rosetta_pbs_batch keeps the extracted ciphertexts (the kN+1 words each
// blind rotation hands to the key switch) in a buffer the library grows with
// cudaMallocAsync when a batch needs more room than it has.  Some callers
// cannot have that happen: a host application whose device memory is owned
// by another allocator (a framework's caching pool that has reserved the
// device), a latency-critical serving loop whose allocation budget is fixed
// after warm-up, or a plugin host that gives plugins no allocation rights.
// This entry point runs the same two kernels with that intermediate buffer
// in a fixed array compiled into the library instead, so it allocates
// nothing; the limit is the array's size.
//
// The array is a file-scope __device__ variable: every GPU that loads the
// library holds it until the process exits, and all calls on a device share
// it.  Host code cannot use its name as a device address, so every call looks
// the address up with cudaGetSymbolAddress on the context's device.  The
// lookup is a host-side table read once the library's device code is loaded
// in the current CUDA context; it is not cached across calls because a
// context that is torn down (cudaDeviceReset) and re-created loads the
// module again at a different address.  The first call on a device, and the
// first after such a reset, loads the module: make it before any stream
// capture.  Calls whose work overlaps on the GPU (for example on two
// streams) race on the array and must be serialised by the caller.  Nothing
// in it has to start at zero: the blind-rotation kernel writes all kN+1
// words of every ciphertext slot it uses before the key switch reads them.
//
// The key switch is the CUDA-core kernel (keyswitch_kernel) at every batch
// size: the tensor-core kernel that rosetta_pbs_batch uses from 256
// ciphertexts on needs digit tiles in a buffer the library allocates.  Both
// give the same words.
#include <cuda_runtime.h>

#include "context.h"
#include "internal.h"

using namespace rosetta;

namespace {

// 16 MiB: 1023 ciphertexts at N = 2048, 511 at N = 4096, 255 at N = 8192.
constexpr size_t kNoallocScratchWords = size_t(2) << 20;
static __device__ __align__(256) uint64_t g_noalloc_scratch[kNoallocScratchWords];

// Device address of g_noalloc_scratch in the current context (the caller
// has made the context's device current).
int noalloc_scratch(uint64_t **out) {
  void *p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
  if (e != cudaSuccess || !p) return ROSETTA_ERR_CUDA;
  *out = static_cast<uint64_t *>(p);
  return ROSETTA_OK;
}

bool on_device(const void *p) {
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

}  // namespace

extern "C" int rosetta_pbs_batch_noalloc(rosetta_ctx *c, const uint64_t *lwe_in, uint32_t batch,
                                         const uint64_t *lut, uint64_t *lwe_out, void *stream) {
  if (!c) return ROSETTA_ERR_INVALID_ARG;
  if (batch == 0) return ROSETTA_OK;
  if (!lwe_in || !lut || !lwe_out) return ROSETTA_ERR_INVALID_ARG;
  if (!c->have_bsk || !c->have_ksk) return ROSETTA_ERR_KEYS_MISSING;
  const size_t kN = static_cast<size_t>(c->prm.glwe_dim) * c->prm.poly_size;
  const size_t n1 = c->prm.lwe_dim + 1;
  if (static_cast<size_t>(batch) * (kN + 1) > kNoallocScratchWords) return ROSETTA_ERR_INVALID_ARG;
  if (c->prm.max_batch && batch > c->prm.max_batch) return ROSETTA_ERR_INVALID_ARG;  // as rosetta_pbs_batch
  const uintptr_t mis = (reinterpret_cast<uintptr_t>(lwe_in) | reinterpret_cast<uintptr_t>(lut) |
                         reinterpret_cast<uintptr_t>(lwe_out)) & 7u;
  if (mis) return ROSETTA_ERR_INVALID_ARG;
  const char *in_b = reinterpret_cast<const char *>(lwe_in), *out_b = reinterpret_cast<const char *>(lwe_out);
  const size_t bytes = static_cast<size_t>(batch) * n1 * 8;
  if (in_b < out_b + bytes && out_b < in_b + bytes) return ROSETTA_ERR_INVALID_ARG;
  if (cudaSetDevice(c->device) != cudaSuccess) return ROSETTA_ERR_CUDA;
  // no staging of host memory here: every buffer must already be on the device
  if (!on_device(lwe_in) || !on_device(lut) || !on_device(lwe_out)) return ROSETTA_ERR_INVALID_ARG;
  uint64_t *big = nullptr;
  const int st = noalloc_scratch(&big);
  if (st != ROSETTA_OK) return st;
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);

  BrArgs a{};
  a.lwe_in = lwe_in;
  a.lut = lut;
  a.lwe_big_out = big;
  br_key_args(c, &a);
  a.n = c->prm.lwe_dim;
  a.level = c->prm.pbs_level;
  a.base_log = c->prm.pbs_base_log;
  a.msg_bits = c->prm.msg_bits;
  a.batch = batch;
  a.num_luts = 1;
  cudaError_t e = launch_blind_rotate(a, c->logN, c->dig16, s);
  if (e != cudaSuccess) return ROSETTA_ERR_CUDA;

  KsArgs k{};
  k.big = big;
  k.out = lwe_out;
  k.ksk = c->d_ksk;
  k.corr = c->d_corr;
  k.batch = batch;
  k.kN = static_cast<uint32_t>(kN);
  k.n = c->prm.lwe_dim;
  k.base_log = c->prm.ks_base_log;
  k.level = c->prm.ks_level;
  e = launch_keyswitch(k, s);
  return e == cudaSuccess ? ROSETTA_OK : ROSETTA_ERR_CUDA;
}
