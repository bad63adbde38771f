/*
 * Seeded synthetic-input generator: Philox4x32-10 (Salmon, Moraes, Dror,
 * Shaw, "Parallel random numbers: as easy as 1, 2, 3", SC'11) followed by the
 * Box-Muller transform.  It produces the random-init weights and the prompt
 * token streams that both the CPU oracle and the CUDA path consume.  Nothing
 * here implements any step of the diffusion model itself.
 *
 * Counter layout: ctr = {blk lo32, blk hi32, stream, 0}, key = {seed lo32,
 * seed hi32}, where blk = element_index / 4 and the (element_index % 4)-th
 * output word belongs to the element.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

#define PHILOX_M0 0xD2511F53u
#define PHILOX_M1 0xCD9E8D57u
#define PHILOX_W0 0x9E3779B9u
#define PHILOX_W1 0xBB67AE85u

void wl_philox4x32_10(const uint32_t ctr_in[4], const uint32_t key_in[2], uint32_t out[4]) {
  uint32_t c0 = ctr_in[0], c1 = ctr_in[1], c2 = ctr_in[2], c3 = ctr_in[3];
  uint32_t k0 = key_in[0], k1 = key_in[1];
  for (int r = 0; r < 10; ++r) {
    if (r > 0) { k0 += PHILOX_W0; k1 += PHILOX_W1; }
    uint64_t p0 = (uint64_t)PHILOX_M0 * c0;
    uint64_t p1 = (uint64_t)PHILOX_M1 * c2;
    uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
    uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
    uint32_t n0 = hi1 ^ c1 ^ k0;
    uint32_t n1 = lo1;
    uint32_t n2 = hi0 ^ c3 ^ k1;
    uint32_t n3 = lo0;
    c0 = n0; c1 = n1; c2 = n2; c3 = n3;
  }
  out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

static void block_words(uint64_t seed, uint32_t stream, uint64_t blk, uint32_t out[4]) {
  uint32_t ctr[4] = {(uint32_t)blk, (uint32_t)(blk >> 32), stream, 0u};
  uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  wl_philox4x32_10(ctr, key, out);
}

/* Raw 32-bit words: out[i] = word (i % 4) of Philox(blk = i / 4). */
void wl_philox_u32(uint64_t seed, uint32_t stream, int64_t n, uint32_t* out) {
  int64_t nblk = (n + 3) / 4;
#pragma omp parallel for schedule(static)
  for (int64_t b = 0; b < nblk; ++b) {
    uint32_t w[4];
    block_words(seed, stream, (uint64_t)b, w);
    for (int j = 0; j < 4; ++j) {
      int64_t i = b * 4 + j;
      if (i < n) out[i] = w[j];
    }
  }
}

/* Words of the blocks first_blk .. first_blk + n_blk - 1: out[4 * j + w] = word w of block first_blk + j. */
void wl_philox_blocks(uint64_t seed, uint32_t stream, uint64_t first_blk, int64_t n_blk, uint32_t* out) {
#pragma omp parallel for schedule(static)
  for (int64_t j = 0; j < n_blk; ++j) block_words(seed, stream, first_blk + (uint64_t)j, out + 4 * j);
}

/* Box-Muller on one Philox block: 4 standard normals. */
static void block_normals(uint64_t seed, uint32_t stream, uint64_t blk, double z[4]) {
  uint32_t w[4];
  block_words(seed, stream, blk, w);
  const double two_pi = 6.283185307179586476925286766559;
  for (int p = 0; p < 2; ++p) {
    double u1 = ((double)(w[2 * p] >> 8) + 1.0) * (1.0 / 16777216.0); /* (0, 1] */
    double u2 = (double)(w[2 * p + 1] >> 8) * (1.0 / 16777216.0);     /* [0, 1) */
    double r = sqrt(-2.0 * log(u1));
    z[2 * p] = r * cos(two_pi * u2);
    z[2 * p + 1] = r * sin(two_pi * u2);
  }
}

static uint16_t f32_to_bf16_rne(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  if ((u & 0x7f800000u) == 0x7f800000u) return (uint16_t)((u >> 16) | ((u & 0xffffu) ? 0x40u : 0u));
  uint32_t lsb = (u >> 16) & 1u;
  u += 0x7fffu + lsb;
  return (uint16_t)(u >> 16);
}

/* out[i] = (float)(mean + std * N_i) */
void wl_normal_f32(uint64_t seed, uint32_t stream, int64_t n, double mean, double std, float* out) {
  int64_t nblk = (n + 3) / 4;
#pragma omp parallel for schedule(static)
  for (int64_t b = 0; b < nblk; ++b) {
    double z[4];
    block_normals(seed, stream, (uint64_t)b, z);
    for (int j = 0; j < 4; ++j) {
      int64_t i = b * 4 + j;
      if (i < n) out[i] = (float)(mean + std * z[j]);
    }
  }
}

/* out[i] = bf16_rne((float)(mean + std * N_i)) as raw bits */
void wl_normal_bf16(uint64_t seed, uint32_t stream, int64_t n, double mean, double std, uint16_t* out) {
  int64_t nblk = (n + 3) / 4;
#pragma omp parallel for schedule(static)
  for (int64_t b = 0; b < nblk; ++b) {
    double z[4];
    block_normals(seed, stream, (uint64_t)b, z);
    for (int j = 0; j < 4; ++j) {
      int64_t i = b * 4 + j;
      if (i < n) out[i] = f32_to_bf16_rne((float)(mean + std * z[j]));
    }
  }
}
