/*
 * rosetta.h — C ABI of the GB300 (sm_103a) batched TFHE programmable
 * bootstrapping library (librosetta.so).
 *
 * What it computes.  The paper (Background, "TFHE Scheme") states the
 * primitive as
 *     [[f(m)]] = TFHE-LUT_f([[m]])
 * for an LWE ciphertext [[m]] in Z_q^{n+1} and a look-up table f whose
 * entries are written into the coefficients of a test polynomial; blind
 * rotation by the encrypted index followed by extraction of the constant
 * term yields a fresh LWE encryption of f(m).  This library evaluates that
 * primitive for a whole batch of independent ciphertexts, with q = 2^64:
 *   1. modulus switch of every word to Z_{2N} (round half up);
 *   2. blind rotation of the test polynomial through n CMux steps, each a
 *      GGSW x GLWE external product (signed gadget decomposition, then exact
 *      negacyclic products in Z_{2^64}[X]/(X^N+1));
 *   3. sample extraction of the constant coefficient (LWE of dimension kN);
 *   4. LWE key switch back to dimension n.
 * Outputs are bit-identical to the plain definition (schoolbook products mod
 * 2^64), not approximations.
 *
 * Word layout.  All ciphertext and key words are uint64 torus elements.
 *   LWE ciphertext   [a_0 .. a_{n-1}, b], phase = b - <a, s>
 *   batch of LWEs    row-major [batch][n+1]
 *   raw BSK          [n][(k+1)*l][k+1][N]; BSK_i is the GGSW of the LWE key
 *                    bit s_i: row r = j*l + (lev-1) is a GLWE encryption of
 *                    0 with s_i * 2^(64 - lev*beta) added to the constant
 *                    coefficient of component j (j = k is the body)
 *   raw KSK          [kN][l_ks][n+1]; row [i][lev] is an LWE encryption under
 *                    the output key of s'_i * 2^(64 - lev*beta_ks), s' the
 *                    extracted GLWE key (s'_{jN+t} = S_j[t])
 *   LUT              2^p torus words lut[m] = Delta * f(m), Delta = 2^(63-p)
 *                    (one padding bit); the test polynomial is
 *                    v[t] = lut[(t + h)/box] for t < N - h and -lut[0] above,
 *                    box = N / 2^p, h = box / 2
 *
 * Pointers and ownership.  The caller owns every buffer it passes and the
 * stream.  Ciphertext and LUT pointers may be device memory or host memory
 * (pinned or pageable); host buffers are staged through library-owned device
 * buffers with copies on the same stream.  Buffers must be 8-byte aligned.
 * Input and output ranges must not overlap.  The library owns the transformed
 * keys, twiddle tables and scratch; rosetta_destroy frees them.
 *
 * Streams and errors.  `stream` is a cudaStream_t passed as void* (NULL =
 * the legacy default stream).  Calls that launch work are asynchronous with
 * respect to the host when every buffer is device memory; with host buffers
 * they return after the copy back has completed.  Every function returns a
 * rosetta_status; argument errors are detected before anything is enqueued.
 * Execution errors surface at rosetta_sync_status or at the next call.
 * No function falls back to the CPU.
 *
 * Threading.  A context may be used from one host thread at a time.  Its
 * scratch buffers (extracted ciphertexts, staging, key-switch digit tiles,
 * lookup intermediates) are shared by its calls, which are ordered only on
 * one stream: work issued through one context on two streams at once must be
 * synchronised by the caller (or use one context per stream).
 */
#ifndef ROSETTA_H
#define ROSETTA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  ROSETTA_OK = 0,
  ROSETTA_ERR_INVALID_ARG = -1,        /* NULL, misaligned, aliasing, bad size, batch too large */
  ROSETTA_ERR_UNSUPPORTED_PARAMS = -2, /* parameter set the kernels do not cover */
  ROSETTA_ERR_KEYS_MISSING = -3,       /* BSK or KSK not uploaded */
  ROSETTA_ERR_CUDA = -4,               /* a CUDA runtime call or launch failed */
  ROSETTA_ERR_OOM = -5,                /* device allocation failed */
  ROSETTA_ERR_TIMEOUT = -6,            /* a bounded device-side wait expired */
  ROSETTA_ERR_BOUNDS = -7              /* a device-side bounds check of a ROSETTA_DEBUG build failed */
} rosetta_status;

typedef struct rosetta_ctx rosetta_ctx; /* opaque, library-owned */

typedef struct {
  uint32_t lwe_dim;      /* n: dimension of input and output LWE ciphertexts */
  uint32_t glwe_dim;     /* k: GLWE dimension (the kernels support k = 1) */
  uint32_t poly_size;    /* N: power of two, 256 .. 8192 */
  uint32_t pbs_base_log; /* beta: PBS gadget base 2^beta, 1 .. 28 */
  uint32_t pbs_level;    /* l: PBS gadget levels, beta*l <= 64 */
  uint32_t ks_base_log;  /* beta_ks: key-switch gadget base, 1 .. 16 */
  uint32_t ks_level;     /* l_ks: key-switch levels, beta_ks*l_ks <= 64 */
  uint32_t msg_bits;     /* p: LUT entries 2^p; N / 2^p must be >= 2 */
  uint32_t max_batch;    /* staging/scratch capacity in ciphertexts; 0 = grow on demand */
} rosetta_params;

/* Create a context on CUDA device `cuda_device` for parameter set *p.
 * Computes the NTT primes' twiddle tables and CRT constants and allocates
 * scratch for p->max_batch ciphertexts.  *out receives the context (NULL on
 * error).  UNSUPPORTED_PARAMS also when the exact external product would
 * not fit the four NTT primes: log2((k+1) l N 2^(beta-1) 2^63) + 1 must not
 * exceed 111 (their product is about 2^111.99); and when one blind-rotation
 * CTA (a quarter of the ring) does not fit the device's shared memory per
 * block: 12N + max(8N, 4.5N per exchange buffer (two for N <= 1024, else
 * one)) + l N x {1 for beta <= 16 | 2} + 2(n+1) bytes, which on a 227 KB
 * device admits at N = 8192, for example, l = 3 with beta <= 16 up to
 * n = 22015, l = 4 or l = 2 with beta > 16 up to n = 17919, and l = 3 with
 * beta > 16 up to n = 9727.  Errors: INVALID_ARG (NULL), UNSUPPORTED_PARAMS,
 * CUDA, OOM. */
int rosetta_params_init(rosetta_ctx **out, const rosetta_params *p, int cuda_device);

/* Number of NTT primes the context's blind rotation computes the external
 * product over: 4 (primes just below 2^28, one CTA per prime in a cluster of
 * four) or 3 (primes just below 2^31, a cluster of three).  The context takes
 * three where (k+1) l N 2^(beta-1) 2^63 <= 0.45 x 2^92.999 (the three primes'
 * product), a three-prime kernel exists (beta <= 16, N = 4096 or 8192,
 * l <= 3) and as many of its CTAs fit one SM's shared memory as of the
 * four-prime kernel's (on a 228 KB SM at N = 4096, l = 2: all n but 10752 to
 * 12799; at N = 8192, l = 3: n <= 15871); e.g. N = 4096, l = 2, beta = 15
 * and N = 8192, l = 3, beta = 14.  Either way the outputs are the same words: the product is
 * exact.  Fixed at rosetta_params_init.  Returns 3 or 4, or INVALID_ARG for a
 * NULL context. */
int rosetta_ntt_primes(const rosetta_ctx *ctx);

/* Upload the raw bootstrapping key (layout above, n_words =
 * n*(k+1)*l*(k+1)*N) and convert it on the device to the transform domain
 * used by the external product (per-prime negacyclic NTT of the centred
 * words, over the context's rosetta_ntt_primes primes).  The source may be host or device memory (src_is_device selects);
 * the caller keeps ownership and may free it after the call returns.  The
 * conversion is stream-ordered on `stream`.  Errors: INVALID_ARG, CUDA, OOM. */
int rosetta_upload_bsk(rosetta_ctx *ctx, const uint64_t *bsk, size_t n_words,
                       int src_is_device, void *stream);

/* Upload the raw key-switching key (n_words = kN*l_ks*(n+1)); same source
 * rules as rosetta_upload_bsk.  Errors: INVALID_ARG, CUDA, OOM. */
int rosetta_upload_ksk(rosetta_ctx *ctx, const uint64_t *ksk, size_t n_words,
                       int src_is_device, void *stream);

/* Programmable bootstrapping of `batch` ciphertexts:
 *   lwe_in  [batch][n+1]  input ciphertexts
 *   lut     [2^p]         torus LUT words (Delta * f(m))
 *   lwe_out [batch][n+1]  PBS outputs (modulus switch, blind rotation,
 *                         sample extraction, key switch)
 * batch == 0 is a no-op returning OK.  Errors: INVALID_ARG, KEYS_MISSING,
 * CUDA, OOM. */
int rosetta_pbs_batch(rosetta_ctx *ctx, const uint64_t *lwe_in, uint32_t batch,
                      const uint64_t *lut, uint64_t *lwe_out, void *stream);

/* The first three steps of rosetta_pbs_batch only: writes the extracted
 * ciphertexts of dimension kN, lwe_big_out [batch][kN+1].  Needs the BSK. */
int rosetta_blind_rotate_extract_batch(rosetta_ctx *ctx, const uint64_t *lwe_in, uint32_t batch,
                                       const uint64_t *lut, uint64_t *lwe_big_out, void *stream);

/* LWE key switch of `batch` ciphertexts of dimension kN, lwe_big_in
 * [batch][kN+1], to dimension n, lwe_out [batch][n+1]:
 *   out = (0, .., 0, b') - sum_i sum_lev d_{i,lev}(a'_i) * KSK[i][lev]
 * with d the signed base-2^beta_ks digits of a'_i rounded to its top
 * beta_ks*l_ks bits.  Needs the KSK.  From 256 ciphertexts on, where the
 * parameters allow exact fp32 sums (beta_ks <= 8 and
 * 2^(beta_ks-1) (2^(64/limbs)-1) kN l_ks < 2^24 for 8 or 16 limbs per key
 * word), the product runs on the tensor cores with a digit scratch of
 * batch (kN l_ks) bf16 words owned by the context; the words are the same
 * either way.  A bounded wait inside that kernel that gives up is reported
 * as TIMEOUT by rosetta_sync_status. */
int rosetta_keyswitch_batch(rosetta_ctx *ctx, const uint64_t *lwe_big_in, uint32_t batch,
                            uint64_t *lwe_out, void *stream);

/* Many LUTs in one launch.  The paper batches independent per-element
 * lookups (Segmented LUT Evaluation, "Multi-Value Batching"), and different
 * nonlinear layers (softmax heads, FFN activations) can share one launch
 * when each ciphertext names its own table: ciphertext b is bootstrapped with
 * LUT luts[lut_index[b]].
 *   luts      [num_luts][2^p] torus words, device memory
 *   lut_index [batch] uint32, device memory, 4-byte aligned
 *   lwe_in / lwe_out as for rosetta_pbs_batch (device or host)
 * The kernel reads luts and lut_index directly.  An index >= num_luts is
 * never followed: that ciphertext uses LUT 0 and the next
 * rosetta_sync_status returns INVALID_ARG.  Errors: INVALID_ARG,
 * KEYS_MISSING, CUDA, OOM. */
int rosetta_pbs_batch_multi_lut(rosetta_ctx *ctx, const uint64_t *lwe_in, uint32_t batch, const uint64_t *luts,
                                uint32_t num_luts, const uint32_t *lut_index, uint64_t *lwe_out, void *stream);

/* Blind rotation of encrypted test polynomials.  The paper's lookup protocol
 * (Cryptographic Lookup Protocol, Steps 2 and 3; Algorithm 1) rotates a
 * per-element RLWE ciphertext of the table, not a public LUT: for each b,
 *   glwe_out[b] = X^{-b~} glwe_in[b] rotated further by X^{a~_i s_i} through
 *                 the n CMux steps, i.e. an encryption of X^{-phi~} M_b where
 *                 glwe_in[b] encrypts M_b and phi~ = b~ - sum a~_i s_i (mod 2N)
 *                 is the modulus-switched phase of lwe_in[b].
 *   lwe_in  [batch][n+1], glwe_in and glwe_out [batch][k+1][N] uint64
 *   (component-major: the k masks, then the body), all device memory.
 * No extraction and no key switch: the result stays a GLWE ciphertext.
 * Needs the BSK.  Errors: INVALID_ARG, KEYS_MISSING, CUDA. */
int rosetta_blind_rotate_glwe_batch(rosetta_ctx *ctx, const uint64_t *lwe_in, uint32_t batch,
                                    const uint64_t *glwe_in, uint64_t *glwe_out, void *stream);

/* Upload the automorphism keys of the RLWE trace (k = 1, N <= 4096).  The
 * paper isolates the constant coefficient of an RLWE ciphertext with a trace
 * (Background, "Scheme Conversion and Other Primitives", RLWE Trace
 * Computation), applied after each blind rotation of its lookup protocol.
 * Step s = 0 .. log2 N - 1 uses X -> X^k, k = 2^(log2 N - s) + 1, and key s:
 * `level` GLWE encryptions under S of sigma_k(S) * 2^(64 - lev*base_log).
 * Raw layout [log2 N][level][2][N] (n_words = log2 N * level * 2 * N);
 * level must be even, 1 <= base_log <= 28, base_log * level <= 64.  Converted
 * on the device like the BSK.  N = 8192 returns UNSUPPORTED_PARAMS: the
 * trace, plaintext-product and lookup kernels keep a whole ciphertext's
 * transform state per cluster in shared memory (about 244 KB per CTA at
 * N = 8192 against the 227 KB a CTA may have); the paper's lookups run on
 * an N_br = 2048 ring.  Errors: INVALID_ARG, UNSUPPORTED_PARAMS, CUDA, OOM. */
int rosetta_upload_trace_keys(rosetta_ctx *ctx, const uint64_t *keys, size_t n_words, uint32_t base_log,
                              uint32_t level, int src_is_device, void *stream);

/* RLWE trace of `batch` GLWE ciphertexts glwe_in [batch][2][N] into glwe_out
 * (same layout, device memory, no overlap): for each step
 *     c <- c + (0, B') - sum_lev D_lev(A') * key_s[lev],  (A', B') = c(X^k)
 * with D the signed gadget digits (base_log, level).  The output encrypts N
 * times the input's constant coefficient (zeros elsewhere): N has no inverse
 * mod 2^64, so callers encode the message at Delta / N.  Exact words (same
 * products mod 2^64 as the definition).  Errors: INVALID_ARG, KEYS_MISSING,
 * CUDA. */
int rosetta_trace_batch(rosetta_ctx *ctx, const uint64_t *glwe_in, uint32_t batch, uint64_t *glwe_out,
                        void *stream);

/* Plaintext x ciphertext polynomial product (k = 1, N <= 4096), the linear
 * mapping of the lookup protocol (Cryptographic Lookup Protocol, Steps 2 and
 * 3: [[t]] = p(X) [[x]] + q(X), [[r_s]] = a_s(X) [[x]] + b_s(X), with the
 * real coefficients encoded as integers by the caller):
 *   glwe_out[b] = (P * A_b, P * B_b + Q)   in Z_{2^64}[X]/(X^N+1)
 *   glwe_in, glwe_out [batch][2][N] uint64, device memory, no overlap
 *   plain_mul [N] int64 P, HOST memory (any value; products are mod 2^64)
 *   plain_add [N] uint64 Q (host or device) or NULL for Q = 0
 * Exact words.  Returns after the work completes.  Errors: INVALID_ARG,
 * UNSUPPORTED_PARAMS, CUDA, OOM. */
int rosetta_plaintext_mul_batch(rosetta_ctx *ctx, const uint64_t *glwe_in, uint32_t batch, const int64_t *plain_mul,
                                const uint64_t *plain_add, uint64_t *glwe_out, void *stream);

/* Tables of one segmented lookup (Segmented LUT Evaluation; Cryptographic
 * Lookup Protocol, Steps 2 and 3), k = 1, N <= 4096, encoded by the caller as
 * integer polynomials (all HOST memory, copied; the call returns when the
 * tables are resident):
 *   p_hat [N] int64, q_hat [N] uint64   -- index polynomials p(X), q(X)
 *   a_hat [n_seg][N] int64, b_hat [n_seg][N] uint64 -- per-segment slope and
 *                                          offset polynomials a_s(X), b_s(X)
 * "Coefficient" s of a polynomial selected by an encrypted index is the box of
 * coefficients a blind rotation by that index can land on: the caller lays
 * out p, q with N / n_seg coefficients per segment and a_s, b_s with
 * N / N_br per interval, each pre-rotated by half a box, the half box below 0
 * negated (as the LUT test polynomial).  n_seg: power of two, 1 .. 256.
 * Replaces any previous tables.  Errors: INVALID_ARG, UNSUPPORTED_PARAMS, CUDA,
 * OOM. */
int rosetta_upload_lookup_table(rosetta_ctx *ctx, uint32_t n_seg, const int64_t *p_hat, const uint64_t *q_hat,
                                const int64_t *a_hat, const uint64_t *b_hat, void *stream);

/* Encrypted segmented lookup f(x) ~ a_SI x + b_SI (Cryptographic Lookup
 * Protocol, Steps 2 and 3; the segment index S comes from the comparisons of
 * Step 1, which are not part of this library):
 *   Step 2: [[t]] = p [[x]] + q; [[I]] = KS(extract(BlindRot([[t]], [[S]])));
 *   Step 3: r_s = Trace(BlindRot(a_s [[x]] + b_s, [[I]])) for every segment s;
 *           R = Box_0 sum_s X^(s N/n_seg) r_s; out = Trace(BlindRot(R, [[S]])).
 *   glwe_x  [batch][2][N] uint64: x in the constant coefficient of the message
 *           (the other message coefficients zero), device memory
 *   lwe_seg [batch][n+1] uint64: LWE of S with Delta = 2^(63 - log2 n_seg), device
 *   glwe_out [batch][2][N] uint64, device, no overlap with the inputs: the phase's
 *           constant coefficient is N^2 (a_SI x + b_SI) in the caller's scale, the
 *           others ~ 0 (each Trace multiplies by N: N has no inverse mod 2^64)
 * Needs the BSK, KSK, trace keys and lookup tables.  Stream-ordered, no host
 * synchronisation.  Per ciphertext: n_seg + 2 plaintext products, n_seg + 2
 * blind rotations, one key switch, n_seg + 1 traces.  Errors: INVALID_ARG,
 * KEYS_MISSING, CUDA, OOM. */
int rosetta_segmented_lookup_batch(rosetta_ctx *ctx, const uint64_t *glwe_x, const uint64_t *lwe_seg, uint32_t batch,
                                   uint64_t *glwe_out, void *stream);

/* Same computation and result as rosetta_pbs_batch, for callers that cannot
 * allocate device memory during the call (their device memory belongs to
 * another allocator, or their serving loop forbids allocation after
 * warm-up).  The paper has no counterpart: this is a deployment variant.
 * The intermediate ciphertexts live in a fixed 16 MiB array compiled into the
 * library (held on every device that loads it until exit) instead of a
 * buffer grown with cudaMallocAsync, so batch * (kN+1) must not exceed
 * 2^21 words (1023 ciphertexts at N = 2048, 255 at N = 8192); larger
 * batches return INVALID_ARG, and so do batches above the context's
 * max_batch, as in rosetta_pbs_batch.  lwe_in, lut and lwe_out must be
 * device memory (no host staging).  Every call looks up the array's device
 * address in the current CUDA context; the first call on a device (and the
 * first after a device reset) loads the library's device code: make it
 * before any stream capture.  The key switch is the CUDA-core kernel at
 * every batch size, because the tensor-core one needs digit tiles in
 * allocated memory (same words).  All calls on a device share the array:
 * calls whose work overlaps on the GPU race and must be serialised by the
 * caller.  Errors: INVALID_ARG, KEYS_MISSING, CUDA. */
int rosetta_pbs_batch_noalloc(rosetta_ctx *ctx, const uint64_t *lwe_in, uint32_t batch,
                              const uint64_t *lut, uint64_t *lwe_out, void *stream);

/* Self-test of the bounded device-side waits (no counterpart in the paper):
 * launches one thread that waits on a barrier nothing completes, gives up
 * after about limit_us microseconds (1 .. 10^6) and raises the context's
 * error flag the way the tensor-core key switch does when one of its waits
 * expires; rosetta_sync_status then returns TIMEOUT once and the context
 * stays usable.  No fault, no hang: the wait is bounded.  Errors:
 * INVALID_ARG, CUDA. */
int rosetta_selftest_wait_timeout(rosetta_ctx *ctx, uint32_t limit_us, void *stream);

/* Self-test of the bounds checks of a library compiled with -DROSETTA_DEBUG
 * (no counterpart in the paper; that build stands in for a memory checker,
 * which this GPU pool does not offer).  The debug kernels compare the key
 * block each CMux step reads with the size of the transformed key and each
 * cluster's ciphertext index with the batch; a failed check skips the access
 * and raises the context's error flag, so rosetta_sync_status returns
 * ROSETTA_ERR_BOUNDS once and the context stays usable (nothing traps).
 * This call blind-rotates one ciphertext, with only its last mask word
 * nonzero, with the key declared one step shorter than it is, so the last
 * step's check fails.  Needs the BSK.  Regular build: UNSUPPORTED_PARAMS.
 * Errors: INVALID_ARG, KEYS_MISSING, CUDA, OOM. */
int rosetta_selftest_bounds(rosetta_ctx *ctx, void *stream);

/* Wait for all work on `stream` and report any deferred execution error
 * (CUDA; TIMEOUT when a bounded wait of the tensor-core key switch gave up;
 * INVALID_ARG for an out-of-range LUT index seen by
 * rosetta_pbs_batch_multi_lut; BOUNDS when a check of a ROSETTA_DEBUG build
 * failed; the flag is cleared once reported).  Returns OK when the stream
 * finished cleanly. */
int rosetta_sync_status(rosetta_ctx *ctx, void *stream);

/* Free everything the context owns.  Waits for the context's device work.
 * NULL is ignored. */
void rosetta_destroy(rosetta_ctx *ctx);

/* Static string naming a status code. */
const char *rosetta_status_string(int status);

#ifdef __cplusplus
}
#endif
#endif /* ROSETTA_H */
