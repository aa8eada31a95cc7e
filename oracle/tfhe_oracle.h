/*
 * Plain CPU oracle for batched TFHE programmable bootstrapping (PBS).
 *
 * TEST INFRASTRUCTURE.  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg may load this library.  The product path
 * (the CUDA library) never calls it and shares no code with it.
 *
 * Everything here is the textbook definition written out, slow on purpose:
 * schoolbook O(N^2) negacyclic products in Z_{2^64}[X]/(X^N+1), gadget
 * decomposition coefficient by coefficient, one CMux at a time.  All words
 * are uint64 with wrap-around arithmetic (the torus Z_q, q = 2^64).
 *
 * The paper (Background, "TFHE Scheme") states PBS as
 *   [[f(m)]] = TFHE-LUT_f([[m]])
 * realised by blind rotation of a test polynomial whose coefficients hold the
 * LUT entries, followed by extraction of the constant term; the remaining
 * conventions (gadget decomposition, GGSW layout, key switching) follow the
 * standard construction the paper cites for PBS (Chillotti et al., TFHE).
 */
#ifndef TFHE_ORACLE_H
#define TFHE_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct {
  uint32_t n;            /* LWE dimension */
  uint32_t k;            /* GLWE dimension */
  uint32_t N;            /* polynomial size */
  uint32_t base_log;     /* PBS gadget: base 2^base_log */
  uint32_t level;        /* PBS gadget: levels */
  uint32_t ks_base_log;  /* key switch gadget base */
  uint32_t ks_level;     /* key switch levels */
  uint32_t msg_bits;     /* p: LUT has 2^p entries, Delta = 2^(63-p) */
} orc_params;

/* ring arithmetic */
void orc_poly_mul_acc(uint64_t *out, const uint64_t *a, const uint64_t *b, uint32_t N);
void orc_poly_mul(uint64_t *out, const uint64_t *a, const uint64_t *b, uint32_t N);
void orc_poly_monomial(uint64_t *out, const uint64_t *a, uint32_t u, uint32_t N);

/* gadget decomposition and modulus switch */
void orc_decompose(uint64_t x, uint32_t base_log, uint32_t level, int64_t *digits);
uint32_t orc_modswitch(uint64_t x, uint32_t log2_2N);

/* encryption (random draws are inputs) */
void orc_lwe_encrypt(uint64_t *out, const uint64_t *s, uint32_t n, uint64_t msg,
                     const uint64_t *mask, uint64_t noise);
uint64_t orc_lwe_phase(const uint64_t *ct, const uint64_t *s, uint32_t n);
void orc_glwe_encrypt(uint64_t *out, const uint64_t *S, uint32_t k, uint32_t N,
                      const uint64_t *msg, const uint64_t *mask, const uint64_t *noise);
void orc_glwe_phase(uint64_t *out, const uint64_t *ct, const uint64_t *S, uint32_t k, uint32_t N);
void orc_ggsw_encrypt(uint64_t *out, const uint64_t *S, uint32_t k, uint32_t N,
                      uint32_t base_log, uint32_t level, uint64_t mu,
                      const uint64_t *mask, const uint64_t *noise);
void orc_bsk_gen(uint64_t *bsk, const orc_params *P, const uint64_t *s_lwe,
                 const uint64_t *S_glwe, const uint64_t *mask, const uint64_t *noise);
void orc_ksk_gen(uint64_t *ksk, const orc_params *P, const uint64_t *s_in,
                 const uint64_t *s_out, const uint64_t *mask, const uint64_t *noise);

/* bootstrapping */
void orc_test_poly(uint64_t *v, const uint64_t *lut, uint32_t msg_bits, uint32_t N);
void orc_external_product(uint64_t *out, const uint64_t *ggsw, const uint64_t *glwe,
                          uint32_t k, uint32_t N, uint32_t base_log, uint32_t level);
void orc_cmux_rotate(uint64_t *acc, const uint64_t *ggsw, uint32_t a_tilde,
                     uint32_t k, uint32_t N, uint32_t base_log, uint32_t level);
void orc_blind_rotate(uint64_t *acc, const orc_params *P, const uint64_t *bsk,
                      const uint64_t *lwe, const uint64_t *lut);
void orc_blind_rotate_glwe(uint64_t *acc, const orc_params *P, const uint64_t *bsk,
                           const uint64_t *lwe, const uint64_t *glwe_in);
void orc_sample_extract(uint64_t *lwe_big, const uint64_t *glwe, uint32_t k, uint32_t N);
void orc_keyswitch(uint64_t *out, const orc_params *P, const uint64_t *ksk, const uint64_t *lwe_big);
void orc_blind_rotate_extract(uint64_t *lwe_big, const orc_params *P, const uint64_t *bsk,
                              const uint64_t *lwe, const uint64_t *lut);
void orc_pbs(uint64_t *out, const orc_params *P, const uint64_t *bsk, const uint64_t *ksk,
             const uint64_t *lwe, const uint64_t *lut);
uint64_t orc_decrypt(const uint64_t *ct, const uint64_t *s, uint32_t n, uint32_t msg_bits);

/* RLWE trace (k = 1) */
void orc_automorphism(uint64_t *out, const uint64_t *a, uint32_t k, uint32_t N);
void orc_auto_key_gen(uint64_t *key, const uint64_t *S, uint32_t N, uint32_t k, uint32_t base_log,
                      uint32_t level, const uint64_t *mask, const uint64_t *noise);
void orc_trace_step(uint64_t *c, const uint64_t *key, uint32_t N, uint32_t k, uint32_t base_log, uint32_t level);
void orc_trace(uint64_t *c, const uint64_t *keys, uint32_t N, uint32_t base_log, uint32_t level);
void orc_plaintext_mul(uint64_t *out, const uint64_t *c, const uint64_t *P, const uint64_t *Qp, uint32_t N);

#ifdef __cplusplus
}
#endif
#endif
