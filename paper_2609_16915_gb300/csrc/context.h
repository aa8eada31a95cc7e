// Layout of the opaque rosetta_ctx handle, shared by the translation units
// that implement the C ABI.
#pragma once
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "rosetta.h"
#include "internal.h"

struct rosetta_ctx {
  rosetta_params prm{};
  int device = 0;
  uint32_t logN = 0;
  bool dig16 = false;
  rosetta::CrtConsts cc{};
  uint2 *d_tw = nullptr;          // [kPrimes][N]
  // the blind rotation's prime set: kPrimes (d_tw, cc) or, where the
  // external-product bound allows, the three 31-bit primes (d_tw31, cc31)
  uint32_t br_primes = rosetta::kPrimes;
  uint2 *d_tw31 = nullptr;        // [kPrimes31][N], or null
  rosetta::CrtConsts cc31{};
  uint32_t *d_bsk = nullptr;      // transform domain over br_primes primes
  size_t bsk_words = 0;           // its size in 32-bit words
  uint64_t *d_ksk = nullptr;      // raw [kN][l_ks][n+1]
  uint64_t *d_corr = nullptr;     // [n+1]
  uint16_t *d_ks_b = nullptr;     // key limb tiles for the tensor-core key switch (null: not exact)
  uint32_t ks_limbs = 0;
  uint64_t *d_ks_a = nullptr;     // digit tiles (scratch), as 64-bit words
  size_t ks_a_cap = 0;
  bool have_bsk = false, have_ksk = false;
  // scratch and staging, sized in ciphertexts
  uint64_t *d_big = nullptr;      // extracted ciphertexts [batch][kN+1]
  size_t big_words_cap = 0;
  uint64_t *d_in = nullptr;       // staging for host inputs
  size_t in_words_cap = 0;
  uint64_t *d_out = nullptr;      // staging for host outputs
  size_t out_words_cap = 0;
  uint64_t *d_lut = nullptr;      // staging for a host LUT  [2^p]
  uint32_t *d_err = nullptr;      // device-side argument error flag (LUT index out of range)
  uint32_t *d_trk = nullptr;      // trace automorphism keys, transform domain
  uint32_t trk_base_log = 0, trk_level = 0;
  bool have_trk = false;
  uint64_t *d_pm_raw = nullptr;   // plaintext-multiply gadget rows, raw [8][2][N]
  uint32_t *d_pm_key = nullptr;   // the same in the transform domain
  uint64_t *d_pm_add = nullptr;   // staged additive plaintext [N]
  // segmented lookup: plaintext polynomials (P, A_0..A_{n_seg-1}, Box_0) as gadget rows in the
  // transform domain [n_seg+2][prime][8][2][N], additive ones (Q, B_0..B_{n_seg-1}) [n_seg+1][N]
  uint32_t *d_lk_key = nullptr;
  uint64_t *d_lk_add = nullptr;
  uint32_t lk_nseg = 0;
  bool have_lk = false;
  uint64_t *d_lk_t = nullptr, *d_lk_u = nullptr, *d_lk_R = nullptr;  // [batch][2][N] each
  size_t lk_t_cap = 0, lk_u_cap = 0, lk_R_cap = 0;
  uint64_t *d_lk_I = nullptr;     // interval-index LWEs [batch][n+1]
  size_t lk_I_cap = 0;
};

// The key, twiddle and CRT fields of a blind rotation over the context's
// bootstrapping key.
inline void br_key_args(const rosetta_ctx *c, rosetta::BrArgs *a) {
  const bool three = c->br_primes == rosetta::kPrimes31;
  a->bsk = c->d_bsk;
  a->bsk_words = c->bsk_words;
  a->primes = c->br_primes;
  a->tw = three ? c->d_tw31 : c->d_tw;
  a->cc = three ? c->cc31 : c->cc;
}
