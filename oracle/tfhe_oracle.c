/*
 * Plain CPU oracle for batched TFHE programmable bootstrapping.
 *
 * TEST INFRASTRUCTURE ONLY (see tfhe_oracle.h).  Slow and literal on purpose:
 * every product is the schoolbook negacyclic convolution, every step is taken
 * in the order the construction states it, and nothing is fused or reordered.
 *
 * Torus: Z_q with q = 2^64; uint64_t arithmetic wraps, which is exactly
 * reduction mod q.
 */
#include "tfhe_oracle.h"

#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------------ */
/* Ring R_{N,q} = Z_q[X]/(X^N + 1)  (Background, "Notation").                */
/* ------------------------------------------------------------------------ */

/* out += a * b in R_{N,q}.  Since X^N = -1, the coefficient t of the product
 * is  sum_{u<=t} a_u b_{t-u}  -  sum_{u>t} a_u b_{N+t-u}. */
void orc_poly_mul_acc(uint64_t *out, const uint64_t *a, const uint64_t *b, uint32_t N) {
  for (uint32_t t = 0; t < N; ++t) {
    uint64_t s = 0;
    for (uint32_t u = 0; u <= t; ++u) s += a[u] * b[t - u];
    for (uint32_t u = t + 1; u < N; ++u) s -= a[u] * b[N + t - u];
    out[t] += s;
  }
}

void orc_poly_mul(uint64_t *out, const uint64_t *a, const uint64_t *b, uint32_t N) {
  memset(out, 0, sizeof(uint64_t) * N);
  orc_poly_mul_acc(out, a, b, N);
}

/* out = X^u * a for u in [0, 2N): coefficient t of a moves to t + u, and each
 * wrap past X^N flips its sign (X^N = -1, X^{2N} = 1).  out must not alias a. */
void orc_poly_monomial(uint64_t *out, const uint64_t *a, uint32_t u, uint32_t N) {
  u %= 2 * N;
  for (uint32_t t = 0; t < N; ++t) {
    uint32_t e = t + u;            /* < 3N */
    uint32_t wraps = e / N;        /* 0, 1 or 2 */
    uint32_t pos = e % N;
    out[pos] = (wraps & 1u) ? (uint64_t)0 - a[t] : a[t];
  }
}

/* ------------------------------------------------------------------------ */
/* Signed gadget decomposition (standard TFHE construction).                 */
/* x is first rounded to its top (level * base_log) bits, c = round(x / 2^(64 */
/* - level*base_log)); then, from the least significant level up, each digit */
/* is the balanced residue of c mod B = 2^base_log, in [-B/2, B/2): a value  */
/* >= B/2 becomes value - B and carries one into the next level.  The final  */
/* carry is dropped (it is a multiple of q).  digits[l-1] is the digit of    */
/* level l, which carries weight 2^(64 - l*base_log), so that                */
/*   sum_l digits[l-1] * 2^(64 - l*base_log) == c * 2^(64 - level*base_log)  */
/* (mod 2^64).  Requires 1 <= base_log <= 31 and level*base_log <= 64.       */
/* ------------------------------------------------------------------------ */
void orc_decompose(uint64_t x, uint32_t base_log, uint32_t level, int64_t *digits) {
  uint32_t bits = base_log * level;
  uint64_t c;
  if (bits >= 64) {
    c = x;
  } else {
    c = (x + ((uint64_t)1 << (63 - bits))) >> (64 - bits);
  }
  const uint64_t B = (uint64_t)1 << base_log;
  for (uint32_t l = level; l >= 1; --l) {
    int64_t d = (int64_t)(c & (B - 1));
    c >>= base_log;
    if ((uint64_t)d >= B / 2) {
      d -= (int64_t)B;
      c += 1;
    }
    digits[l - 1] = d;
  }
}

/* Modulus switch of a torus word to Z_{2N}: round(x * 2N / 2^64) mod 2N, with
 * ties rounded up.  Named "ModSwitch" in the paper's conversion pipeline
 * (Segmented LUT Evaluation, Pipeline Integration). */
uint32_t orc_modswitch(uint64_t x, uint32_t log2_2N) {
  uint32_t sh = 64 - log2_2N;
  uint64_t r = (x + ((uint64_t)1 << (sh - 1))) >> sh;
  return (uint32_t)(r & (((uint64_t)1 << log2_2N) - 1));
}

/* ------------------------------------------------------------------------ */
/* Encryption (Background, "TFHE Scheme": [[m]] in Z_q^{n+1}).                */
/* Convention: b = <a, s> + m + e, phase = b - <a, s>.                        */
/* ------------------------------------------------------------------------ */
void orc_lwe_encrypt(uint64_t *out, const uint64_t *s, uint32_t n, uint64_t msg,
                     const uint64_t *mask, uint64_t noise) {
  uint64_t b = 0;
  for (uint32_t i = 0; i < n; ++i) {
    out[i] = mask[i];
    b += mask[i] * s[i];
  }
  out[n] = b + msg + noise;
}

uint64_t orc_lwe_phase(const uint64_t *ct, const uint64_t *s, uint32_t n) {
  uint64_t acc = ct[n];
  for (uint32_t i = 0; i < n; ++i) acc -= ct[i] * s[i];
  return acc;
}

/* Decrypt: round(phase / Delta) mod 2^(p+1), Delta = 2^(63-p) (one padding bit). */
uint64_t orc_decrypt(const uint64_t *ct, const uint64_t *s, uint32_t n, uint32_t msg_bits) {
  uint64_t ph = orc_lwe_phase(ct, s, n);
  uint32_t sh = 63 - msg_bits;
  uint64_t r = (ph + ((uint64_t)1 << (sh - 1))) >> sh;
  return r & (((uint64_t)1 << (msg_bits + 1)) - 1);
}

/* GLWE (RLWE when k = 1, Background "FHE Schemes"): ct = (A_0..A_{k-1}, B),
 * B = sum_j A_j * S_j + M + E.  msg may be NULL (encryption of zero). */
void orc_glwe_encrypt(uint64_t *out, const uint64_t *S, uint32_t k, uint32_t N,
                      const uint64_t *msg, const uint64_t *mask, const uint64_t *noise) {
  uint64_t *B = out + (size_t)k * N;
  memset(B, 0, sizeof(uint64_t) * N);
  for (uint32_t j = 0; j < k; ++j) {
    memcpy(out + (size_t)j * N, mask + (size_t)j * N, sizeof(uint64_t) * N);
    orc_poly_mul_acc(B, mask + (size_t)j * N, S + (size_t)j * N, N);
  }
  for (uint32_t t = 0; t < N; ++t) B[t] += (msg ? msg[t] : 0) + noise[t];
}

/* phase = B - sum_j A_j * S_j */
void orc_glwe_phase(uint64_t *out, const uint64_t *ct, const uint64_t *S, uint32_t k, uint32_t N) {
  uint64_t *tmp = (uint64_t *)calloc(N, sizeof(uint64_t));
  for (uint32_t j = 0; j < k; ++j) orc_poly_mul_acc(tmp, ct + (size_t)j * N, S + (size_t)j * N, N);
  for (uint32_t t = 0; t < N; ++t) out[t] = ct[(size_t)k * N + t] - tmp[t];
  free(tmp);
}

/* GGSW encryption of the constant polynomial mu.  Row r = j*level + (l-1)
 * (j in [0,k] the component, l in [1,level]) is a fresh GLWE encryption of 0
 * with mu * 2^(64 - l*base_log) added to the constant coefficient of its
 * component j.  Layout out[r][c][t], r < (k+1)level, c < k+1, t < N.
 * mask: [(k+1)level][k][N], noise: [(k+1)level][N]. */
void orc_ggsw_encrypt(uint64_t *out, const uint64_t *S, uint32_t k, uint32_t N,
                      uint32_t base_log, uint32_t level, uint64_t mu,
                      const uint64_t *mask, const uint64_t *noise) {
  const size_t row_words = (size_t)(k + 1) * N;
  for (uint32_t j = 0; j <= k; ++j) {
    for (uint32_t l = 1; l <= level; ++l) {
      uint32_t r = j * level + (l - 1);
      uint64_t *row = out + (size_t)r * row_words;
      orc_glwe_encrypt(row, S, k, N, NULL, mask + (size_t)r * k * N, noise + (size_t)r * N);
      row[(size_t)j * N] += mu << (64 - l * base_log);
    }
  }
}

/* Bootstrapping key: the n GGSW encryptions of the LWE secret bits s_i under
 * the GLWE key.  Layout [n][(k+1)level][k+1][N]. */
void orc_bsk_gen(uint64_t *bsk, const orc_params *P, const uint64_t *s_lwe,
                 const uint64_t *S_glwe, const uint64_t *mask, const uint64_t *noise) {
  const uint32_t rows = (P->k + 1) * P->level;
  const size_t ggsw_words = (size_t)rows * (P->k + 1) * P->N;
  for (uint32_t i = 0; i < P->n; ++i) {
    orc_ggsw_encrypt(bsk + i * ggsw_words, S_glwe, P->k, P->N, P->base_log, P->level, s_lwe[i],
                     mask + (size_t)i * rows * P->k * P->N, noise + (size_t)i * rows * P->N);
  }
}

/* Key-switching key from the extracted key s_in (length kN) to the LWE key
 * s_out (length n): row [i][l] is an LWE encryption under s_out of
 * s_in[i] * 2^(64 - l*ks_base_log).  Layout [kN][ks_level][n+1].
 * mask: [kN][ks_level][n], noise: [kN][ks_level]. */
void orc_ksk_gen(uint64_t *ksk, const orc_params *P, const uint64_t *s_in,
                 const uint64_t *s_out, const uint64_t *mask, const uint64_t *noise) {
  const uint32_t kN = P->k * P->N;
  for (uint32_t i = 0; i < kN; ++i) {
    for (uint32_t l = 1; l <= P->ks_level; ++l) {
      size_t r = (size_t)i * P->ks_level + (l - 1);
      orc_lwe_encrypt(ksk + r * (P->n + 1), s_out, P->n, s_in[i] << (64 - l * P->ks_base_log),
                      mask + r * P->n, noise[r]);
    }
  }
}

/* ------------------------------------------------------------------------ */
/* Programmable bootstrapping (Background, "TFHE Scheme", PBS).               */
/* ------------------------------------------------------------------------ */

/* Test polynomial: the LUT entries laid out as coefficients, each entry
 * repeated over a box of N/2^p coefficients so that the rotation amount,
 * which carries noise, only needs to land inside the right box.  The boxes
 * are shifted down by half a box (h = box/2): v[t] = lut[(t + h) / box] for
 * t < N - h, and the last h coefficients hold -lut[0], the negacyclic image of
 * entry 0.  Rotating left by phi (multiplying by X^{-phi}) then brings
 * lut[round(phi / box)] to the constant coefficient, the left rotation of the
 * paper's figure (LUT (6,7,3,5), m = 2 gives 3). */
void orc_test_poly(uint64_t *v, const uint64_t *lut, uint32_t msg_bits, uint32_t N) {
  const uint32_t box = N >> msg_bits;
  const uint32_t h = box / 2;
  for (uint32_t t = 0; t < N; ++t) {
    v[t] = (t < N - h) ? lut[(t + h) / box] : (uint64_t)0 - lut[0];
  }
}

/* External product GGSW (x) GLWE: each component C_j of the GLWE is split
 * into `level` digit polynomials D_{j,l} (gadget decomposition of every
 * coefficient), and out_c = sum_{j,l} D_{j,l} * GGSW[j*level + l - 1][c]. */
void orc_external_product(uint64_t *out, const uint64_t *ggsw, const uint64_t *glwe,
                          uint32_t k, uint32_t N, uint32_t base_log, uint32_t level) {
  const size_t row_words = (size_t)(k + 1) * N;
  uint64_t *dig = (uint64_t *)malloc(sizeof(uint64_t) * N);
  int64_t d[64];
  memset(out, 0, sizeof(uint64_t) * row_words);
  for (uint32_t j = 0; j <= k; ++j) {
    for (uint32_t l = 1; l <= level; ++l) {
      for (uint32_t t = 0; t < N; ++t) {
        orc_decompose(glwe[(size_t)j * N + t], base_log, level, d);
        dig[t] = (uint64_t)d[l - 1];
      }
      const uint64_t *row = ggsw + (size_t)(j * level + (l - 1)) * row_words;
      for (uint32_t c = 0; c <= k; ++c) orc_poly_mul_acc(out + (size_t)c * N, dig, row + (size_t)c * N, N);
    }
  }
  free(dig);
}

/* One CMux step of blind rotation: ACC <- ACC + GGSW (x) (X^{a} * ACC - ACC).
 * With GGSW encrypting a bit s, this rotates ACC by X^{a*s}. */
void orc_cmux_rotate(uint64_t *acc, const uint64_t *ggsw, uint32_t a_tilde,
                     uint32_t k, uint32_t N, uint32_t base_log, uint32_t level) {
  const size_t words = (size_t)(k + 1) * N;
  uint64_t *diff = (uint64_t *)malloc(sizeof(uint64_t) * words);
  uint64_t *prod = (uint64_t *)malloc(sizeof(uint64_t) * words);
  for (uint32_t c = 0; c <= k; ++c) {
    orc_poly_monomial(diff + (size_t)c * N, acc + (size_t)c * N, a_tilde, N);
    for (uint32_t t = 0; t < N; ++t) diff[(size_t)c * N + t] -= acc[(size_t)c * N + t];
  }
  orc_external_product(prod, ggsw, diff, k, N, base_log, level);
  for (size_t t = 0; t < words; ++t) acc[t] += prod[t];
  free(diff);
  free(prod);
}

static uint32_t log2_u32(uint32_t x) {
  uint32_t r = 0;
  while ((1u << r) < x) ++r;
  return r;
}

/* The n CMux steps of blind rotation on an accumulator already initialised
 * to X^{-b~} times the test polynomial (public or encrypted). */
static void cmux_steps(uint64_t *acc, const orc_params *P, const uint64_t *bsk, const uint64_t *lwe,
                       uint32_t log2_2N) {
  const size_t ggsw_words = (size_t)(P->k + 1) * P->level * (P->k + 1) * P->N;
  for (uint32_t i = 0; i < P->n; ++i) {
    uint32_t a_tilde = orc_modswitch(lwe[i], log2_2N);
    if (a_tilde == 0) continue;
    orc_cmux_rotate(acc, bsk + i * ggsw_words, a_tilde, P->k, P->N, P->base_log, P->level);
  }
}

/* Blind rotation: modulus-switch the LWE to Z_{2N} (a~_i, b~), start from the
 * trivial GLWE (0, X^{-b~} * v), then for i = 0..n-1 rotate by X^{a~_i s_i}
 * through the CMux with BSK_i.  The result encrypts X^{-phi~} * v with
 * phi~ = b~ - sum a~_i s_i.  A step with a~_i = 0 is skipped: the difference
 * X^0 * ACC - ACC is zero, its decomposition is zero and the step adds 0. */
void orc_blind_rotate(uint64_t *acc, const orc_params *P, const uint64_t *bsk,
                      const uint64_t *lwe, const uint64_t *lut) {
  const uint32_t N = P->N, k = P->k;
  const uint32_t log2_2N = log2_u32(2 * N);
  const size_t ggsw_words = (size_t)(k + 1) * P->level * (k + 1) * N;
  uint64_t *v = (uint64_t *)malloc(sizeof(uint64_t) * N);
  orc_test_poly(v, lut, P->msg_bits, N);
  memset(acc, 0, sizeof(uint64_t) * (size_t)(k + 1) * N);
  uint32_t b_tilde = orc_modswitch(lwe[P->n], log2_2N);
  orc_poly_monomial(acc + (size_t)k * N, v, (2 * N - b_tilde) % (2 * N), N);
  (void)ggsw_words;
  cmux_steps(acc, P, bsk, lwe, log2_2N);
  free(v);
}

/* Blind rotation of an encrypted test polynomial (the lookup protocol's
 * BlindRot of a per-element RLWE ciphertext, Cryptographic Lookup Protocol
 * Steps 2-3): the accumulator starts as X^{-b~} times the input GLWE
 * (every component), then the same n CMux steps. */
void orc_blind_rotate_glwe(uint64_t *acc, const orc_params *P, const uint64_t *bsk, const uint64_t *lwe,
                           const uint64_t *glwe_in) {
  const uint32_t N = P->N;
  const uint32_t log2_2N = log2_u32(2 * N);
  const uint32_t b_tilde = orc_modswitch(lwe[P->n], log2_2N);
  for (uint32_t c = 0; c <= P->k; ++c)
    orc_poly_monomial(acc + (size_t)c * N, glwe_in + (size_t)c * N, (2 * N - b_tilde) % (2 * N), N);
  cmux_steps(acc, P, bsk, lwe, log2_2N);
}

/* Sample extraction of the constant coefficient (Background, "LWE Extract"):
 * a'_{jN} = A_j[0], a'_{jN+t} = -A_j[N-t] (t >= 1), b' = B[0]; the result is
 * an LWE ciphertext of dimension kN under the key s'_{jN+t} = S_j[t]. */
void orc_sample_extract(uint64_t *lwe_big, const uint64_t *glwe, uint32_t k, uint32_t N) {
  for (uint32_t j = 0; j < k; ++j) {
    const uint64_t *A = glwe + (size_t)j * N;
    lwe_big[(size_t)j * N] = A[0];
    for (uint32_t t = 1; t < N; ++t) lwe_big[(size_t)j * N + t] = (uint64_t)0 - A[N - t];
  }
  lwe_big[(size_t)k * N] = glwe[(size_t)k * N];
}

/* LWE key switch from dimension kN back to n: out = (0,...,0,b') -
 * sum_i sum_l d_{i,l} * KSK[i][l], d_{i,l} the gadget digits of a'_i. */
void orc_keyswitch(uint64_t *out, const orc_params *P, const uint64_t *ksk, const uint64_t *lwe_big) {
  const uint32_t kN = P->k * P->N, n = P->n;
  int64_t d[64];
  memset(out, 0, sizeof(uint64_t) * (n + 1));
  out[n] = lwe_big[kN];
  for (uint32_t i = 0; i < kN; ++i) {
    orc_decompose(lwe_big[i], P->ks_base_log, P->ks_level, d);
    for (uint32_t l = 1; l <= P->ks_level; ++l) {
      const uint64_t *row = ksk + ((size_t)i * P->ks_level + (l - 1)) * (n + 1);
      const uint64_t dl = (uint64_t)d[l - 1];
      for (uint32_t o = 0; o <= n; ++o) out[o] -= dl * row[o];
    }
  }
}

/* ------------------------------------------------------------------------ */
/* RLWE trace (Background, "Scheme Conversion and Other Primitives", RLWE    */
/* Trace Computation: a logarithmic sequence of Galois automorphisms and     */
/* additions leaves only the constant term).  k = 1.                          */
/* ------------------------------------------------------------------------ */

/* out = a(X^k) in R_{N,q} for odd k: coefficient t moves to t k mod 2N, with
 * a sign flip when that exponent lies in [N, 2N).  out must not alias a. */
void orc_automorphism(uint64_t *out, const uint64_t *a, uint32_t k, uint32_t N) {
  for (uint32_t t = 0; t < N; ++t) {
    uint64_t e = ((uint64_t)t * k) % (2 * (uint64_t)N);
    if (e < N) out[e] = a[t];
    else out[e - N] = (uint64_t)0 - a[t];
  }
}

/* Automorphism key for X -> X^k: row l (l = 1..level) is a GLWE encryption
 * under S of sigma_k(S) * 2^(64 - l*base_log).  Layout [level][2][N].
 * mask: [level][N], noise: [level][N]. */
void orc_auto_key_gen(uint64_t *key, const uint64_t *S, uint32_t N, uint32_t k, uint32_t base_log,
                      uint32_t level, const uint64_t *mask, const uint64_t *noise) {
  uint64_t *sig = (uint64_t *)malloc(sizeof(uint64_t) * N);
  uint64_t *msg = (uint64_t *)malloc(sizeof(uint64_t) * N);
  orc_automorphism(sig, S, k, N);
  for (uint32_t l = 1; l <= level; ++l) {
    for (uint32_t t = 0; t < N; ++t) msg[t] = sig[t] << (64 - l * base_log);
    orc_glwe_encrypt(key + (size_t)(l - 1) * 2 * N, S, 1, N, msg, mask + (size_t)(l - 1) * N,
                     noise + (size_t)(l - 1) * N);
  }
  free(sig);
  free(msg);
}

/* c <- c + KS(sigma_k(c)) with KS(A', B') = (0, B') - sum_l D_l(A') * key[l]:
 * the automorphed ciphertext is an encryption under sigma_k(S); the key
 * switch brings it back under S, and the sum doubles the coefficients the
 * automorphism fixes and cancels the ones it negates. */
void orc_trace_step(uint64_t *c, const uint64_t *key, uint32_t N, uint32_t k, uint32_t base_log, uint32_t level) {
  uint64_t *sA = (uint64_t *)malloc(sizeof(uint64_t) * N);
  uint64_t *sB = (uint64_t *)malloc(sizeof(uint64_t) * N);
  uint64_t *dig = (uint64_t *)malloc(sizeof(uint64_t) * N);
  uint64_t *prod = (uint64_t *)calloc(2 * (size_t)N, sizeof(uint64_t));
  int64_t d[64];
  orc_automorphism(sA, c, k, N);
  orc_automorphism(sB, c + N, k, N);
  for (uint32_t l = 1; l <= level; ++l) {
    for (uint32_t t = 0; t < N; ++t) {
      orc_decompose(sA[t], base_log, level, d);
      dig[t] = (uint64_t)d[l - 1];
    }
    for (uint32_t comp = 0; comp < 2; ++comp)
      orc_poly_mul_acc(prod + (size_t)comp * N, dig, key + ((size_t)(l - 1) * 2 + comp) * N, N);
  }
  for (uint32_t t = 0; t < N; ++t) {
    c[t] -= prod[t];
    c[N + t] += sB[t] - prod[N + t];
  }
  free(sA);
  free(sB);
  free(dig);
  free(prod);
}

/* Trace to the constant coefficient: for j = log2 N down to 1, apply the
 * step with k = 2^j + 1 (key j-1 of keys [log2 N][level][2][N]: keys[0] for
 * k = N + 1, ..., keys[log2 N - 1] for k = 3).  The phase becomes N times the
 * constant coefficient of the input phase, zeros elsewhere; on the torus
 * Z_{2^64} N has no inverse, so the factor N stays (the caller encodes the
 * message at scale Delta / N). */
void orc_trace(uint64_t *c, const uint64_t *keys, uint32_t N, uint32_t base_log, uint32_t level) {
  uint32_t logN = 0;
  while ((1u << logN) < N) ++logN;
  for (uint32_t s = 0; s < logN; ++s) {
    uint32_t k = (1u << (logN - s)) + 1;
    orc_trace_step(c, keys + (size_t)s * level * 2 * N, N, k, base_log, level);
  }
}

/* Plaintext x ciphertext product (k = 1): (P * A, P * B + Q), the linear
 * mapping of the lookup protocol.  Q may be NULL. */
void orc_plaintext_mul(uint64_t *out, const uint64_t *c, const uint64_t *P, const uint64_t *Qp, uint32_t N) {
  orc_poly_mul(out, P, c, N);
  orc_poly_mul(out + N, P, c + N, N);
  if (Qp)
    for (uint32_t t = 0; t < N; ++t) out[N + t] += Qp[t];
}

void orc_blind_rotate_extract(uint64_t *lwe_big, const orc_params *P, const uint64_t *bsk,
                              const uint64_t *lwe, const uint64_t *lut) {
  uint64_t *acc = (uint64_t *)malloc(sizeof(uint64_t) * (size_t)(P->k + 1) * P->N);
  orc_blind_rotate(acc, P, bsk, lwe, lut);
  orc_sample_extract(lwe_big, acc, P->k, P->N);
  free(acc);
}

/* PBS = modulus switch -> blind rotation -> sample extraction -> key switch. */
void orc_pbs(uint64_t *out, const orc_params *P, const uint64_t *bsk, const uint64_t *ksk,
             const uint64_t *lwe, const uint64_t *lut) {
  uint64_t *big = (uint64_t *)malloc(sizeof(uint64_t) * ((size_t)P->k * P->N + 1));
  orc_blind_rotate_extract(big, P, bsk, lwe, lut);
  orc_keyswitch(out, P, ksk, big);
  free(big);
}
