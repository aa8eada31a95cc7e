/* A C program that uses librosetta through include/rosetta.h only (no CUDA
 * headers, no Python): reads a parameter set, keys, a LUT and LWE
 * ciphertexts from a file, bootstraps them with host buffers and writes the
 * results.  The GPU test compares the output with the CPU oracle.
 *
 * Input file (little-endian): 9 uint32 (rosetta_params fields in order),
 * uint32 batch, then uint64 words: BSK, KSK, LUT (2^p), LWE [batch][n+1].
 * Output file: uint64 [batch][n+1]. */
#include <stdio.h>
#include <stdlib.h>

#include "rosetta.h"

static int read_words(FILE *f, uint64_t *dst, size_t n) { return fread(dst, sizeof(uint64_t), n, f) == n ? 0 : -1; }

int main(int argc, char **argv) {
  if (argc != 3) {
    fprintf(stderr, "usage: %s input output\n", argv[0]);
    return 2;
  }
  FILE *f = fopen(argv[1], "rb");
  if (!f) return 2;
  uint32_t h[10];
  if (fread(h, sizeof(uint32_t), 10, f) != 10) return 2;
  rosetta_params p = {h[0], h[1], h[2], h[3], h[4], h[5], h[6], h[7], h[8]};
  const uint32_t batch = h[9];
  const size_t n1 = (size_t)p.lwe_dim + 1;
  const size_t bsk_words = (size_t)p.lwe_dim * (p.glwe_dim + 1) * p.pbs_level * (p.glwe_dim + 1) * p.poly_size;
  const size_t ksk_words = (size_t)p.glwe_dim * p.poly_size * p.ks_level * n1;
  const size_t lut_words = (size_t)1 << p.msg_bits;
  uint64_t *bsk = malloc(bsk_words * 8), *ksk = malloc(ksk_words * 8), *lut = malloc(lut_words * 8);
  uint64_t *in = malloc(batch * n1 * 8), *out = malloc(batch * n1 * 8);
  if (!bsk || !ksk || !lut || !in || !out) return 2;
  if (read_words(f, bsk, bsk_words) || read_words(f, ksk, ksk_words) || read_words(f, lut, lut_words) ||
      read_words(f, in, batch * n1))
    return 2;
  fclose(f);

  rosetta_ctx *ctx = NULL;
  int st = rosetta_params_init(&ctx, &p, 0);
  if (st == ROSETTA_OK) st = rosetta_upload_bsk(ctx, bsk, bsk_words, 0, NULL);
  if (st == ROSETTA_OK) st = rosetta_upload_ksk(ctx, ksk, ksk_words, 0, NULL);
  if (st == ROSETTA_OK) st = rosetta_pbs_batch(ctx, in, batch, lut, out, NULL);
  if (st == ROSETTA_OK) st = rosetta_sync_status(ctx, NULL);
  if (st != ROSETTA_OK) {
    fprintf(stderr, "rosetta: %s (%d)\n", rosetta_status_string(st), st);
    rosetta_destroy(ctx);
    return 1;
  }
  rosetta_destroy(ctx);
  FILE *g = fopen(argv[2], "wb");
  if (!g || fwrite(out, sizeof(uint64_t), batch * n1, g) != batch * n1) return 2;
  fclose(g);
  free(bsk);
  free(ksk);
  free(lut);
  free(in);
  free(out);
  return 0;
}
