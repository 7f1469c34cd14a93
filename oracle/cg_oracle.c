/*
 * cg_oracle.c -- plain, slow, fp64 CPU oracle for the canary-trap hot path.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product library calls, links or
 * includes this file; only the tests, the package's smoke check and the CPU
 * baseline leg of the benchmark load it.  It shares no header, helper, table
 * or constant generator with the CUDA path.
 *
 * What it computes (arxiv 2607.19490, "Integrity of peer-to-peer distributed
 * LLM inference under malicious nodes"):
 *   - the synthetic hop-local pipeline: fp32 reference a (Eq. 1 stand-in),
 *     benign live h = a + delta (Eq. 2), tampered live h = tau(a) (Eq. 3 and
 *     the three tamper strategies of Sec. 3.2), rounded to fp16 (Sec. 3.3);
 *   - the relative-L2 mismatch m = ||h - a||_F / ||a||_F (Eq. 4), the cosine
 *     mismatch 1 - h.a/(||h|| ||a||) (cosine ablation, Sec. 4.4) and the
 *     max-abs deviation;
 *   - the per-canary AUROC (Eq. 5) by brute force over every
 *     (malicious, benign) pair, ties counted as one half (Mann-Whitney), and
 *     its mean over canaries (Eq. 6);
 *   - the scrambled-label negative control (Sec. 4.5).
 * Random numbers come from Philox4x32-10 as defined by Salmon, Moraes, Dror
 * and Shaw, "Parallel Random Numbers: As Easy as 1, 2, 3" (SC'11), normals
 * from the Box-Muller transform, bounded integers from Lemire's
 * multiply-shift method with rejection ("Fast Random Integer Generation in an
 * Interval", ACM TOMACS 2019).
 *
 * Every floating-point step is carried out in double precision.  Build with
 * -ffp-contract=off so that no multiply-add is fused on any host.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* ------------------------------------------------------------------------ */
/* Status codes returned by the oracle entry points.                         */
enum { OR_OK = 0, OR_BAD_ARG = 1, OR_NAN_SCORE = 2, OR_NO_MEMORY = 3 };

/* Noise models and tamper kinds (numbering matches the public API enums;   */
/* the values are restated here, not included).                             */
enum { OR_NOISE_MULT = 0, OR_NOISE_PAPER = 1 };
enum { OR_TAMPER_ADDITIVE = 0, OR_TAMPER_SIGNFLIP_CHANNELS = 1,
       OR_TAMPER_SIGNFLIP_FULL = 2, OR_TAMPER_SCALE = 3 };

/* Counter layout of every draw: (c0, c1, c2, c3) =                        */
/*   element streams: (block q of the segment, segment s*N + n,             */
/*                     4 * config_id + stream, 0)                           */
/*   auxiliary words: (word index / 4, (purpose << 24) | sub,               */
/*                     4 * config_id + OR_STREAM_AUX, 0)                    */
/* so config_id must stay below 2^30.  c3 is 0 for every draw of the live   */
/* pipeline; an independent benign recompute r (the redundant-recompute      */
/* ceiling and the noisy-reference ablation, Sec. 4.4-4.5) draws its noise   */
/* with c3 = r, so replica 0 is the live draw itself.                        */
enum { OR_STREAM_REF = 0, OR_STREAM_NOISE = 1, OR_STREAM_TAMPER = 2,
       OR_STREAM_AUX = 3 };
enum { OR_AUX_OUTLIER = 1, OR_AUX_SHARD_SIGMA = 2, OR_AUX_FLIP = 3,
       OR_AUX_CONTROL = 4, OR_AUX_RANDOM = 5 };

/* ------------------------------------------------------------------------ */
/* Philox4x32-10 (SC'11, Sec. 5): ten rounds of the two-multiply S-box with   */
/* the Weyl-sequence key schedule.                                           */
void or_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2],
                      uint32_t out[4]) {
  const uint32_t M0 = 0xD2511F53u, M1 = 0xCD9E8D57u;
  const uint32_t W0 = 0x9E3779B9u, W1 = 0xBB67AE85u;
  uint32_t x0 = ctr[0], x1 = ctr[1], x2 = ctr[2], x3 = ctr[3];
  uint32_t k0 = key[0], k1 = key[1];
  for (int round = 0; round < 10; ++round) {
    uint64_t p0 = (uint64_t)M0 * (uint64_t)x0;
    uint64_t p1 = (uint64_t)M1 * (uint64_t)x2;
    uint32_t y0 = (uint32_t)(p1 >> 32) ^ x1 ^ k0;
    uint32_t y1 = (uint32_t)p1;
    uint32_t y2 = (uint32_t)(p0 >> 32) ^ x3 ^ k1;
    uint32_t y3 = (uint32_t)p0;
    x0 = y0; x1 = y1; x2 = y2; x3 = y3;
    k0 += W0;
    k1 += W1;
  }
  out[0] = x0; out[1] = x1; out[2] = x2; out[3] = x3;
}

static void seed_to_key(uint64_t seed, uint32_t key[2]) {
  key[0] = (uint32_t)(seed & 0xFFFFFFFFu);
  key[1] = (uint32_t)(seed >> 32);
}

/* Raw words of blocks first_block .. first_block + n_blocks - 1 with the     */
/* counter (block, c1, c2, c3); 4 words per block, block-major.              */
void or_philox_words(uint64_t seed, uint32_t c1, uint32_t c2, uint32_t c3,
                     uint32_t first_block, uint32_t n_blocks, uint32_t *out) {
  uint32_t key[2];
  seed_to_key(seed, key);
  for (uint32_t i = 0; i < n_blocks; ++i) {
    uint32_t ctr[4] = {first_block + i, c1, c2, c3};
    or_philox4x32_10(ctr, key, out + 4 * (size_t)i);
  }
}

/* ------------------------------------------------------------------------ */
/* Uniforms and the Box-Muller transform.                                    */
/*   u1 = ((x0 >> 8) + 1) * 2^-24 in (0, 1]   (never 0, so log is finite)    */
/*   u2 =  (x1 >> 8)      * 2^-24 in [0, 1)                                  */
/*   z0 = sqrt(-2 ln u1) cos(2 pi u2),  z1 = sqrt(-2 ln u1) sin(2 pi u2)     */
void or_box_muller(uint32_t x0, uint32_t x1, double *z0, double *z1) {
  const double two_pi = 6.283185307179586476925286766559;
  double u1 = ((double)(x0 >> 8) + 1.0) * 0x1p-24;
  double u2 = (double)(x1 >> 8) * 0x1p-24;
  double r = sqrt(-2.0 * log(u1));
  double theta = two_pi * u2;
  *z0 = r * cos(theta);
  *z1 = r * sin(theta);
}

/* The transform over word pairs: pair i = (words[2i], words[2i+1]). */
void or_box_muller_pairs(const uint32_t *words, uint64_t n_pairs, double *out) {
  for (uint64_t i = 0; i < n_pairs; ++i)
    or_box_muller(words[2 * i], words[2 * i + 1], out + 2 * i, out + 2 * i + 1);
}

/* Normals of blocks [first_block, first_block + n_blocks): 4 per block,     */
/* (x0, x1) -> elements 0, 1 and (x2, x3) -> elements 2, 3.                  */
void or_philox_normals(uint64_t seed, uint32_t c1, uint32_t c2, uint32_t c3,
                       uint32_t first_block, uint32_t n_blocks, double *out) {
  uint32_t key[2];
  seed_to_key(seed, key);
  for (uint32_t i = 0; i < n_blocks; ++i) {
    uint32_t ctr[4] = {first_block + i, c1, c2, c3};
    uint32_t w[4];
    or_philox4x32_10(ctr, key, w);
    or_box_muller(w[0], w[1], out + 4 * (size_t)i + 0, out + 4 * (size_t)i + 1);
    or_box_muller(w[2], w[3], out + 4 * (size_t)i + 2, out + 4 * (size_t)i + 3);
  }
}

/* ------------------------------------------------------------------------ */
/* Auxiliary word stream and Lemire's bounded draw.                          */
typedef struct {
  uint32_t key[2];
  uint32_t c1, c2;
  uint64_t next;       /* index of the next word in the stream */
  uint64_t cached;     /* block index held in blk, or UINT64_MAX */
  uint32_t blk[4];
} or_words;

static void words_init(or_words *w, uint64_t seed, uint32_t purpose,
                       uint32_t sub, uint32_t config_id) {
  seed_to_key(seed, w->key);
  w->c1 = (purpose << 24) | (sub & 0x00FFFFFFu);
  w->c2 = 4u * config_id + OR_STREAM_AUX;
  w->next = 0;
  w->cached = UINT64_MAX;
}

static uint32_t words_next(or_words *w) {
  uint64_t q = w->next >> 2;
  if (q != w->cached) {
    uint32_t ctr[4] = {(uint32_t)q, w->c1, w->c2, 0u};
    or_philox4x32_10(ctr, w->key, w->blk);
    w->cached = q;
  }
  uint32_t x = w->blk[w->next & 3];
  w->next += 1;
  return x;
}

/* Uniform integer in [0, n), n >= 1: multiply-shift with rejection of the */
/* low-word range below (2^32 - n) mod n (Lemire 2019).                     */
static uint32_t words_bounded(or_words *w, uint32_t n) {
  uint64_t m = (uint64_t)words_next(w) * (uint64_t)n;
  uint32_t low = (uint32_t)m;
  if (low < n) {
    uint32_t threshold = (uint32_t)(0u - n) % n;
    while (low < threshold) {
      m = (uint64_t)words_next(w) * (uint64_t)n;
      low = (uint32_t)m;
    }
  }
  return (uint32_t)(m >> 32);
}

/* k distinct values of [0, n) in draw order; duplicates are redrawn.        */
static int draw_distinct(uint64_t seed, uint32_t purpose, uint32_t sub,
                         uint32_t config_id, uint32_t n, uint32_t k,
                         uint32_t *out) {
  if (k > n) return OR_BAD_ARG;
  unsigned char *taken = (unsigned char *)calloc(n ? n : 1, 1);
  if (!taken) return OR_NO_MEMORY;
  or_words w;
  words_init(&w, seed, purpose, sub, config_id);
  uint32_t got = 0;
  while (got < k) {
    uint32_t v = words_bounded(&w, n);
    if (taken[v]) continue;
    taken[v] = 1;
    out[got++] = v;
  }
  free(taken);
  return OR_OK;
}

/* Exposed for tests: the first `count` bounded draws of an aux stream.      */
void or_aux_bounded(uint64_t seed, uint32_t purpose, uint32_t sub,
                    uint32_t config_id, uint32_t n, uint32_t count,
                    uint32_t *out) {
  or_words w;
  words_init(&w, seed, purpose, sub, config_id);
  for (uint32_t i = 0; i < count; ++i) out[i] = words_bounded(&w, n);
}

/* ------------------------------------------------------------------------ */
/* IEEE binary16 conversion, round to nearest, ties to even, subnormals      */
/* kept, overflow to infinity.                                               */
uint16_t or_half_from_double(double x) {
  uint16_t sign = signbit(x) ? 0x8000u : 0u;
  if (isnan(x)) return (uint16_t)(sign | 0x7E00u);
  double ax = fabs(x);
  /* 65520 is halfway between 65504 (largest finite, odd mantissa) and 2^16. */
  if (ax >= 65520.0) return (uint16_t)(sign | 0x7C00u);
  if (ax < 0x1p-14) {
    /* subnormal (or zero): value = q * 2^-24 with integer q in [0, 1024]   */
    double q = nearbyint(ax * 0x1p24);   /* exact scaling; ties to even */
    return (uint16_t)(sign | (uint16_t)q); /* q == 1024 is the smallest normal */
  }
  int ex;
  double f = frexp(ax, &ex);             /* ax = f * 2^ex, f in [0.5, 1) */
  int e = ex - 1;                        /* ax = (2f) * 2^e, 2f in [1, 2) */
  double mant = nearbyint((2.0 * f - 1.0) * 1024.0);
  if (mant == 1024.0) { mant = 0.0; e += 1; }
  if (e > 15) return (uint16_t)(sign | 0x7C00u);
  return (uint16_t)(sign | (uint16_t)((e + 15) << 10) | (uint16_t)mant);
}

double or_half_to_double(uint16_t h) {
  int sign = (h >> 15) & 1;
  int e = (h >> 10) & 0x1F;
  int m = h & 0x3FF;
  double v;
  if (e == 0) v = ldexp((double)m, -24);
  else if (e == 31) v = m ? NAN : INFINITY;
  else v = ldexp(1.0 + m / 1024.0, e - 15);
  return sign ? -v : v;
}

/* ------------------------------------------------------------------------ */
/* Pipeline description (the oracle's own; parameters are the binary32      */
/* values the API carries, widened to double).                               */
typedef struct {
  uint32_t n_shards, hidden, n_canaries, tokens; /* k, d, n, T */
  const int32_t *malicious;                      /* 0-based stage ids */
  uint32_t n_malicious;                          /* c = |M| */
  int32_t noise;                                 /* OR_NOISE_* */
  double benign_sigma;                           /* sigma_hw (Eq. 2) */
  double shard_sigma_lognormal;                  /* 0: one sigma for all */
  uint32_t n_outlier;
  double outlier_scale;
  int32_t tamper;                                /* OR_TAMPER_* */
  double tamper_param;                           /* eps | fraction | factor */
  uint64_t seed;
  uint32_t config_id;
} or_desc;

typedef struct {
  uint32_t *outlier;     /* n_outlier channel ids */
  double *shard_sigma;   /* per stage sigma */
  unsigned char *is_mal; /* per stage */
  unsigned char *flip;   /* [S][d] channel flip flags (channel tamper) */
} or_tables;

static uint32_t flip_count(double p, uint32_t d) {
  double r = floor(p * (double)d + 0.5);
  uint32_t n = (r < 1.0) ? 1u : (uint32_t)r;
  return n > d ? d : n;
}

static int check_desc(const or_desc *D) {
  if (!D || D->n_shards < 1 || D->hidden < 1 || D->n_canaries < 1 ||
      D->tokens < 1)
    return OR_BAD_ARG;
  if (D->n_malicious >= D->n_shards) return OR_BAD_ARG;
  if (D->config_id >= (1u << 30)) return OR_BAD_ARG;
  if (D->n_malicious && !D->malicious) return OR_BAD_ARG;
  if (D->n_outlier > D->hidden) return OR_BAD_ARG;
  if (D->noise != OR_NOISE_MULT && D->noise != OR_NOISE_PAPER) return OR_BAD_ARG;
  if (D->tamper < OR_TAMPER_ADDITIVE || D->tamper > OR_TAMPER_SCALE)
    return OR_BAD_ARG;
  if (D->tamper == OR_TAMPER_SIGNFLIP_CHANNELS &&
      !(D->tamper_param > 0.0 && D->tamper_param <= 1.0))
    return OR_BAD_ARG;
  for (uint32_t i = 0; i < D->n_malicious; ++i) {
    if (D->malicious[i] < 0 || (uint32_t)D->malicious[i] >= D->n_shards)
      return OR_BAD_ARG;
    for (uint32_t j = 0; j < i; ++j)
      if (D->malicious[j] == D->malicious[i]) return OR_BAD_ARG;
  }
  return OR_OK;
}

static void free_tables(or_tables *t) {
  free(t->outlier); free(t->shard_sigma); free(t->is_mal); free(t->flip);
  memset(t, 0, sizeof(*t));
}

/* Per-configuration draws: outlier channels, per-stage sigma, flip sets.    */
static int build_tables(const or_desc *D, or_tables *t) {
  memset(t, 0, sizeof(*t));
  uint32_t S = D->n_shards, d = D->hidden;
  t->outlier = (uint32_t *)calloc(D->n_outlier ? D->n_outlier : 1, 4);
  t->shard_sigma = (double *)calloc(S, sizeof(double));
  t->is_mal = (unsigned char *)calloc(S, 1);
  t->flip = (unsigned char *)calloc((size_t)S * d, 1);
  if (!t->outlier || !t->shard_sigma || !t->is_mal || !t->flip) {
    free_tables(t);
    return OR_NO_MEMORY;
  }
  int st = draw_distinct(D->seed, OR_AUX_OUTLIER, 0, D->config_id, d,
                         D->n_outlier, t->outlier);
  if (st) { free_tables(t); return st; }
  for (uint32_t s = 0; s < S; ++s) {
    if (D->shard_sigma_lognormal > 0.0) {
      or_words w;
      words_init(&w, D->seed, OR_AUX_SHARD_SIGMA, s, D->config_id);
      uint32_t x0 = words_next(&w), x1 = words_next(&w);
      double z0, z1;
      or_box_muller(x0, x1, &z0, &z1);
      t->shard_sigma[s] = D->benign_sigma * exp(D->shard_sigma_lognormal * z0);
    } else {
      t->shard_sigma[s] = D->benign_sigma;
    }
  }
  for (uint32_t i = 0; i < D->n_malicious; ++i) {
    uint32_t s = (uint32_t)D->malicious[i];
    t->is_mal[s] = 1;
    if (D->tamper == OR_TAMPER_SIGNFLIP_CHANNELS) {
      uint32_t nf = flip_count(D->tamper_param, d);
      uint32_t *ch = (uint32_t *)malloc(nf * sizeof(uint32_t));
      if (!ch) { free_tables(t); return OR_NO_MEMORY; }
      st = draw_distinct(D->seed, OR_AUX_FLIP, s, D->config_id, d, nf, ch);
      if (st) { free(ch); free_tables(t); return st; }
      for (uint32_t j = 0; j < nf; ++j) t->flip[(size_t)s * d + ch[j]] = 1;
      free(ch);
    }
  }
  return OR_OK;
}

/* Exposed for tests: the drawn tables of one configuration.                 */
int or_config_tables(const or_desc *D, uint32_t *outlier, double *shard_sigma,
                     unsigned char *flip /* [S][d] */) {
  int st = check_desc(D);
  if (st) return st;
  or_tables t;
  st = build_tables(D, &t);
  if (st) return st;
  if (outlier && D->n_outlier)
    memcpy(outlier, t.outlier, D->n_outlier * sizeof(uint32_t));
  if (shard_sigma) memcpy(shard_sigma, t.shard_sigma, D->n_shards * sizeof(double));
  if (flip) memcpy(flip, t.flip, (size_t)D->n_shards * D->hidden);
  free_tables(&t);
  return OR_OK;
}

/* The normal of element e of segment seg on stream `stream`.                */
static double element_normal_r(const uint32_t key[2], uint32_t seg,
                               uint32_t config_id, uint32_t stream, uint32_t c3,
                               uint64_t e) {
  uint32_t ctr[4] = {(uint32_t)(e >> 2), seg, 4u * config_id + stream, c3};
  uint32_t w[4];
  or_philox4x32_10(ctr, key, w);
  double z[4];
  or_box_muller(w[0], w[1], &z[0], &z[1]);
  or_box_muller(w[2], w[3], &z[2], &z[3]);
  return z[e & 3];
}

static double element_normal(const uint32_t key[2], uint32_t seg,
                             uint32_t config_id, uint32_t stream, uint64_t e) {
  return element_normal_r(key, seg, config_id, stream, 0u, e);
}

/* Benign output of stage s on segment (s, n) with the noise of replica r   */
/* (Eq. 2): MULT a (1 + sigma_s z), PAPER a + sigma_s mu z.                  */
static void benign_values(const or_desc *D, const or_tables *t, uint32_t s,
                          uint32_t seg, const double *a, uint64_t L,
                          uint32_t replica, double *live, double *coef_out) {
  uint32_t key[2];
  seed_to_key(D->seed, key);
  double sig = t->shard_sigma[s];
  double coef = 0.0;
  if (D->noise == OR_NOISE_MULT) {
    for (uint64_t e = 0; e < L; ++e) {
      double z = element_normal_r(key, seg, D->config_id, OR_STREAM_NOISE, replica, e);
      live[e] = a[e] * (1.0 + sig * z);
    }
  } else {
    double l1 = 0.0;
    for (uint64_t e = 0; e < L; ++e) l1 += fabs(a[e]);
    double mu = l1 / (double)L;
    coef = sig * mu;
    for (uint64_t e = 0; e < L; ++e) {
      double z = element_normal_r(key, seg, D->config_id, OR_STREAM_NOISE, replica, e);
      live[e] = a[e] + coef * z;
    }
  }
  if (coef_out) *coef_out = coef;
}

/* One (stage s, canary n) segment of T*d elements, token-major.             */
/*   refs: fp32 reference a (synthetic stand-in for Eq. 1)                   */
/*   pre : live value before fp16 rounding, double (may be NULL)             */
/*   acts: fp16 live h (Eq. 2 benign / Eq. 3 tampered), binary16 bits        */
/*   coef: per-segment scalar: sigma_s * mu (PAPER noise), the additive      */
/*         tamper's eps*||a||/||g||, else 0 (may be NULL)                    */
static int segment(const or_desc *D, const or_tables *t, uint32_t s,
                   uint32_t n, float *refs, double *pre, uint16_t *acts,
                   double *coef_out) {
  const uint32_t d = D->hidden;
  const uint64_t L = (uint64_t)D->tokens * d;
  const uint32_t seg = s * D->n_canaries + n;
  uint32_t key[2];
  seed_to_key(D->seed, key);

  double *a = (double *)malloc(L * sizeof(double));
  double *live = (double *)malloc(L * sizeof(double));
  if (!a || !live) { free(a); free(live); return OR_NO_MEMORY; }

  /* reference: a = z_ref * (outlier_scale on an outlier channel, else 1),   */
  /* stored in fp32; everything downstream uses the stored fp32 value.       */
  for (uint64_t e = 0; e < L; ++e) {
    uint32_t c = (uint32_t)(e % d);
    double scale = 1.0;
    for (uint32_t j = 0; j < D->n_outlier; ++j)
      if (t->outlier[j] == c) scale = D->outlier_scale;
    double z = element_normal(key, seg, D->config_id, OR_STREAM_REF, e);
    float af = (float)(z * scale);
    a[e] = (double)af;
    if (refs) refs[e] = af;
  }

  double coef = 0.0;
  if (!t->is_mal[s]) {
    benign_values(D, t, s, seg, a, L, 0u, live, &coef);
  } else if (D->tamper == OR_TAMPER_ADDITIVE) {
    /* Gaussian tamper: tau(v) = v + eps ||v||_F g / ||g||_F */
    double aa = 0.0, gg = 0.0;
    for (uint64_t e = 0; e < L; ++e) {
      double g = element_normal(key, seg, D->config_id, OR_STREAM_TAMPER, e);
      aa += a[e] * a[e];
      gg += g * g;
    }
    coef = (gg > 0.0) ? D->tamper_param * sqrt(aa) / sqrt(gg) : 0.0;
    for (uint64_t e = 0; e < L; ++e) {
      double g = element_normal(key, seg, D->config_id, OR_STREAM_TAMPER, e);
      live[e] = a[e] + coef * g;
    }
  } else if (D->tamper == OR_TAMPER_SIGNFLIP_CHANNELS) {
    for (uint64_t e = 0; e < L; ++e) {
      uint32_t c = (uint32_t)(e % d);
      live[e] = t->flip[(size_t)s * d + c] ? -a[e] : a[e];
    }
  } else if (D->tamper == OR_TAMPER_SIGNFLIP_FULL) {
    for (uint64_t e = 0; e < L; ++e) live[e] = -a[e];     /* tau(v) = -v */
  } else {                                                /* rescale */
    for (uint64_t e = 0; e < L; ++e) live[e] = D->tamper_param * a[e];
  }

  for (uint64_t e = 0; e < L; ++e) {
    if (pre) pre[e] = live[e];
    if (acts) acts[e] = or_half_from_double(live[e]);
  }
  if (coef_out) *coef_out = coef;
  free(a);
  free(live);
  return OR_OK;
}

/* One segment, for sampled checks at sizes too large to generate whole.    */
int or_generate_segment(const or_desc *D, uint32_t s, uint32_t n, float *refs,
                        double *pre, uint16_t *acts, double *coef) {
  int st = check_desc(D);
  if (st) return st;
  if (s >= D->n_shards || n >= D->n_canaries) return OR_BAD_ARG;
  or_tables t;
  st = build_tables(D, &t);
  if (st) return st;
  st = segment(D, &t, s, n, refs, pre, acts, coef);
  free_tables(&t);
  return st;
}

/* Whole pipeline: acts/refs [S][N][T][d], labels [N][S] (1 = malicious).    */
int or_generate_pipeline(const or_desc *D, uint16_t *acts, float *refs,
                         int8_t *labels, int n_threads) {
  int st = check_desc(D);
  if (st) return st;
  or_tables t;
  st = build_tables(D, &t);
  if (st) return st;
  const uint32_t S = D->n_shards, N = D->n_canaries;
  const uint64_t L = (uint64_t)D->tokens * D->hidden;
  int err = OR_OK;
#ifdef _OPENMP
  if (n_threads > 0) omp_set_num_threads(n_threads);
#pragma omp parallel for schedule(dynamic, 1)
#endif
  for (int64_t q = 0; q < (int64_t)S * N; ++q) {
    uint32_t s = (uint32_t)(q / N), n = (uint32_t)(q % N);
    size_t off = (size_t)q * L;
    int e = segment(D, &t, s, n, refs ? refs + off : NULL, NULL,
                    acts ? acts + off : NULL, NULL);
    if (e) {
#ifdef _OPENMP
#pragma omp critical
#endif
      err = e;
    }
  }
  if (labels)
    for (uint32_t n = 0; n < N; ++n)
      for (uint32_t s = 0; s < S; ++s)
        labels[(size_t)n * S + s] = (int8_t)t.is_mal[s];
  free_tables(&t);
  (void)n_threads;
  return err;
}

/* Segments first .. first + count - 1 of the pipeline (segment q = s*N+n),  */
/* written one after another to acts/refs [count][T*d]: the same values as   */
/* the matching slice of or_generate_pipeline, for pipelines too large to    */
/* hold whole on the host (one stage at a time).  coef [count] (may be NULL) */
/* receives each segment's scalar as or_generate_segment returns it.         */
int or_generate_segments(const or_desc *D, uint64_t first, uint64_t count,
                         uint16_t *acts, float *refs, double *coef,
                         int n_threads) {
  int st = check_desc(D);
  if (st) return st;
  const uint64_t n_seg = (uint64_t)D->n_shards * D->n_canaries;
  if (first > n_seg || count > n_seg - first) return OR_BAD_ARG;
  or_tables t;
  st = build_tables(D, &t);
  if (st) return st;
  const uint32_t N = D->n_canaries;
  const uint64_t L = (uint64_t)D->tokens * D->hidden;
  int err = OR_OK;
#ifdef _OPENMP
  if (n_threads > 0) omp_set_num_threads(n_threads);
#pragma omp parallel for schedule(dynamic, 1)
#endif
  for (int64_t i = 0; i < (int64_t)count; ++i) {
    const uint64_t q = first + (uint64_t)i;
    uint32_t s = (uint32_t)(q / N), n = (uint32_t)(q % N);
    size_t off = (size_t)i * L;
    int e = segment(D, &t, s, n, refs ? refs + off : NULL, NULL,
                    acts ? acts + off : NULL, coef ? coef + i : NULL);
    if (e) {
#ifdef _OPENMP
#pragma omp critical
#endif
      err = e;
    }
  }
  free_tables(&t);
  (void)n_threads;
  return err;
}

/* Propagating pipeline (Eq. 2's recursion h_i = f_i(h_{i-1}) + delta_i     */
/* with the block's response to its input linearised as                     */
/*     f_i(h_{i-1}) = a_i + gain * (h_{i-1} - a_{i-1}),                     */
/* h_{-1} = a_{-1}, i.e. the first stage sees the exact embedding).  With   */
/* v_i = f_i(h_{i-1}):                                                       */
/*   benign    h_i = fp16(v_i + sigma_i mu_i z), mu_i = ||v_i||_1 / (T d)    */
/*             (MULT: fp16(v_i (1 + sigma_i z)))                            */
/*   malicious h_i = fp16(tau(v_i)) (Eq. 3 with v = f(h_{i*-1}), Sec. 3.2)   */
/* Stages are produced in order, each from the previous stage's fp16 live   */
/* values; gain = 0 is the hop-local pipeline of or_generate_pipeline.      */
int or_generate_propagating(const or_desc *D, double gain, uint16_t *acts,
                            float *refs, int n_threads) {
  int st = check_desc(D);
  if (st) return st;
  or_tables t;
  st = build_tables(D, &t);
  if (st) return st;
  const uint32_t S = D->n_shards, N = D->n_canaries, d = D->hidden;
  const uint64_t L = (uint64_t)D->tokens * d;
  int err = OR_OK;
#ifdef _OPENMP
  if (n_threads > 0) omp_set_num_threads(n_threads);
#pragma omp parallel for schedule(dynamic, 1)
#endif
  for (int64_t nn = 0; nn < (int64_t)N; ++nn) {
    const uint32_t n = (uint32_t)nn;
    uint32_t key[2];
    seed_to_key(D->seed, key);
    double *a = (double *)malloc(L * sizeof(double));
    double *v = (double *)malloc(L * sizeof(double));
    double *dev = (double *)calloc(L, sizeof(double));   /* h_{i-1} - a_{i-1} */
    if (!a || !v || !dev) {
      free(a); free(v); free(dev);
#ifdef _OPENMP
#pragma omp critical
#endif
      err = OR_NO_MEMORY;
      continue;
    }
    for (uint32_t s = 0; s < S; ++s) {
      const uint32_t seg = s * N + n;
      const size_t off = (size_t)seg * L;
      for (uint64_t e = 0; e < L; ++e) {
        uint32_t c = (uint32_t)(e % d);
        double scale = 1.0;
        for (uint32_t j = 0; j < D->n_outlier; ++j)
          if (t.outlier[j] == c) scale = D->outlier_scale;
        float af = (float)(element_normal(key, seg, D->config_id, OR_STREAM_REF, e) * scale);
        a[e] = (double)af;
        if (refs) refs[off + e] = af;
        v[e] = a[e] + gain * dev[e];
      }
      double *live = dev;   /* reuse: live values of this stage */
      if (!t.is_mal[s]) {
        double sig = t.shard_sigma[s];
        if (D->noise == OR_NOISE_MULT) {
          for (uint64_t e = 0; e < L; ++e)
            live[e] = v[e] * (1.0 + sig * element_normal(key, seg, D->config_id,
                                                          OR_STREAM_NOISE, e));
        } else {
          double l1 = 0.0;
          for (uint64_t e = 0; e < L; ++e) l1 += fabs(v[e]);
          double coef = sig * (l1 / (double)L);
          for (uint64_t e = 0; e < L; ++e)
            live[e] = v[e] + coef * element_normal(key, seg, D->config_id,
                                                   OR_STREAM_NOISE, e);
        }
      } else if (D->tamper == OR_TAMPER_ADDITIVE) {
        double vv = 0.0, gg = 0.0;
        for (uint64_t e = 0; e < L; ++e) {
          double g = element_normal(key, seg, D->config_id, OR_STREAM_TAMPER, e);
          vv += v[e] * v[e];
          gg += g * g;
        }
        double coef = (gg > 0.0) ? D->tamper_param * sqrt(vv) / sqrt(gg) : 0.0;
        for (uint64_t e = 0; e < L; ++e)
          live[e] = v[e] + coef * element_normal(key, seg, D->config_id,
                                                 OR_STREAM_TAMPER, e);
      } else if (D->tamper == OR_TAMPER_SIGNFLIP_CHANNELS) {
        for (uint64_t e = 0; e < L; ++e)
          live[e] = t.flip[(size_t)s * d + (uint32_t)(e % d)] ? -v[e] : v[e];
      } else if (D->tamper == OR_TAMPER_SIGNFLIP_FULL) {
        for (uint64_t e = 0; e < L; ++e) live[e] = -v[e];
      } else {
        for (uint64_t e = 0; e < L; ++e) live[e] = D->tamper_param * v[e];
      }
      for (uint64_t e = 0; e < L; ++e) {
        uint16_t hb = or_half_from_double(live[e]);
        if (acts) acts[off + e] = hb;
        dev[e] = or_half_to_double(hb) - a[e];
      }
    }
    free(a); free(v); free(dev);
  }
  free_tables(&t);
  (void)n_threads;
  return err;
}

/* An independent benign recompute of every stage (Sec. 4.5, redundant-     */
/* recompute ceiling; Sec. 4.4, noisy reference): the benign output of each */
/* stage, malicious ones included, with the noise of replica r, rounded to  */
/* fp16 and stored as fp32 [S][N][T][d].  Replica 0 is the live draw.       */
int or_generate_recompute(const or_desc *D, uint32_t replica, float *out,
                          int n_threads) {
  int st = check_desc(D);
  if (st) return st;
  or_tables t;
  st = build_tables(D, &t);
  if (st) return st;
  const uint32_t S = D->n_shards, N = D->n_canaries, d = D->hidden;
  const uint64_t L = (uint64_t)D->tokens * d;
  int err = OR_OK;
#ifdef _OPENMP
  if (n_threads > 0) omp_set_num_threads(n_threads);
#pragma omp parallel for schedule(dynamic, 1)
#endif
  for (int64_t q = 0; q < (int64_t)S * N; ++q) {
    uint32_t s = (uint32_t)(q / N), n = (uint32_t)(q % N);
    uint32_t seg = s * N + n;
    uint32_t key[2];
    seed_to_key(D->seed, key);
    double *a = (double *)malloc(L * sizeof(double));
    double *h = (double *)malloc(L * sizeof(double));
    if (!a || !h) {
      free(a); free(h);
#ifdef _OPENMP
#pragma omp critical
#endif
      err = OR_NO_MEMORY;
      continue;
    }
    for (uint64_t e = 0; e < L; ++e) {
      uint32_t c = (uint32_t)(e % d);
      double scale = 1.0;
      for (uint32_t j = 0; j < D->n_outlier; ++j)
        if (t.outlier[j] == c) scale = D->outlier_scale;
      a[e] = (double)(float)(element_normal(key, seg, D->config_id,
                                            OR_STREAM_REF, e) * scale);
    }
    benign_values(D, &t, s, seg, a, L, replica, h, NULL);
    for (uint64_t e = 0; e < L; ++e)
      out[(size_t)q * L + e] = (float)or_half_to_double(or_half_from_double(h[e]));
    free(a);
    free(h);
  }
  free_tables(&t);
  (void)n_threads;
  return err;
}

/* Random baseline (Sec. 4.5): every score replaced by Uniform(0, 1).        */
/* scores[c][n][s] = (x >> 8) 2^-24, x = word s of aux stream (RANDOM, sub   */
/* = canary n) with config id config_id0 + c.                                */
void or_random_scores(uint64_t seed, uint32_t config_id0, uint32_t C,
                      uint32_t N, uint32_t S, float *out) {
  for (uint32_t c = 0; c < C; ++c)
    for (uint32_t n = 0; n < N; ++n) {
      or_words w;
      words_init(&w, seed, OR_AUX_RANDOM, n, config_id0 + c);
      for (uint32_t s = 0; s < S; ++s)
        out[((size_t)c * N + n) * S + s] =
            (float)((double)(words_next(&w) >> 8) * 0x1p-24);
    }
}

/* ------------------------------------------------------------------------ */
/* Drift scores of one segment of L elements (h = fp16 live, a = fp32 ref). */
/*   rel_l2  = ||h - a|| / ||a||                          (Eq. 4)            */
/*   max_abs = max |h - a|  (NaN elements are skipped, like C's fmax)        */
/*   cos_dev = 1 - h.a / (||h|| ||a||)                    (cosine ablation)  */
/* cos_dev is evaluated as (1/2) || h/||h|| - a/||a|| ||^2, which equals     */
/* 1 - cos for unit vectors and is a sum of non-negative terms (no           */
/* cancellation).  Edge cases: ||a|| = 0 gives rel_l2 = 0 if h = a else      */
/* +inf; cos_dev is 0 when either norm is 0.                                 */
void or_drift_segment(const uint16_t *acts, const float *refs, uint64_t L,
                      double out[3], double sums[4]) {
  double D = 0.0, A = 0.0, H = 0.0, M = 0.0;
  for (uint64_t e = 0; e < L; ++e) {
    double h = or_half_to_double(acts[e]);
    double a = (double)refs[e];
    double diff = h - a;
    D += diff * diff;
    A += a * a;
    H += h * h;
    M = fmax(M, fabs(diff));
  }
  double rel = (A > 0.0) ? sqrt(D / A) : (D == 0.0 ? 0.0 : INFINITY);
  if (isnan(D) || isnan(A)) rel = NAN;
  double cosd = 0.0;
  if (isnan(H) || isnan(A)) {
    cosd = NAN;
  } else if (H > 0.0 && A > 0.0) {
    double nh = sqrt(H), na = sqrt(A), acc = 0.0;
    for (uint64_t e = 0; e < L; ++e) {
      double u = or_half_to_double(acts[e]) / nh - (double)refs[e] / na;
      acc += u * u;
    }
    cosd = 0.5 * acc;
  }
  out[0] = rel;
  out[1] = M;
  out[2] = cosd;
  if (sums) { sums[0] = D; sums[1] = A; sums[2] = H; sums[3] = M; }
}

/* acts/refs [S][N][L]; scores[stat * stat_stride + n * S + s].             */
void or_drift_scores(const uint16_t *acts, const float *refs, uint32_t S,
                     uint32_t N, uint64_t L, double *scores,
                     uint64_t stat_stride, int n_threads) {
#ifdef _OPENMP
  if (n_threads > 0) omp_set_num_threads(n_threads);
#pragma omp parallel for schedule(dynamic, 1)
#endif
  for (int64_t q = 0; q < (int64_t)S * N; ++q) {
    uint32_t s = (uint32_t)(q / N), n = (uint32_t)(q % N);
    double out[3];
    or_drift_segment(acts + (size_t)q * L, refs + (size_t)q * L, L, out, NULL);
    for (int k = 0; k < 3; ++k)
      scores[(size_t)k * stat_stride + (size_t)n * S + s] = out[k];
  }
  (void)n_threads;
}

/* ------------------------------------------------------------------------ */
/* Mann-Whitney counts and AUROC (Eq. 5, Eq. 6).                             */
/* scores, labels: [C][N][S]; labels 1 = malicious, 0 = benign, -1 = left    */
/* out.  For each (config, canary):                                          */
/*   gt = #{(i, j): label_i = 1, label_j = 0, m_i > m_j}                     */
/*   eq = #{(i, j): label_i = 1, label_j = 0, m_i = m_j}                     */
/*   u2 = 2 gt + eq   (twice the Mann-Whitney U, ties counted as one half)   */
/*   pairs = c_t * b_t                                                       */
/* A^(t) = u2 / (2 pairs) is Eq. 5 with ties as halves; canaries with no     */
/* pair are skipped.  A-hat (Eq. 6) is the mean of A^(t) over the remaining  */
/* canaries: when every one has the same pair count P it is evaluated as     */
/* sum(u2) / (2 P N_valid), one division of exact integers; otherwise the    */
/* A^(t) are added in canary order and the sum divided by N_valid.           */
/* Returns OR_NAN_SCORE if a labelled score is NaN.                          */
int or_auroc(const float *scores, const int8_t *labels, uint32_t C,
             uint32_t N, uint32_t S, int64_t *u2, int64_t *gt, int64_t *eq,
             int64_t *pairs, double *auroc) {
  int status = OR_OK;
  for (uint32_t c = 0; c < C; ++c) {
    int64_t total_u2 = 0, common = -1, n_valid = 0;
    int uniform = 1;
    for (uint32_t n = 0; n < N; ++n) {
      const float *m = scores + ((size_t)c * N + n) * S;
      const int8_t *l = labels + ((size_t)c * N + n) * S;
      int64_t g = 0, e = 0, nm = 0, nb = 0;
      for (uint32_t i = 0; i < S; ++i) {
        if (l[i] == 1) nm++;
        if (l[i] == 0) nb++;
        if ((l[i] == 1 || l[i] == 0) && isnan(m[i])) status = OR_NAN_SCORE;
      }
      for (uint32_t i = 0; i < S; ++i) {
        if (l[i] != 1) continue;
        for (uint32_t j = 0; j < S; ++j) {
          if (l[j] != 0) continue;
          if (m[i] > m[j]) g++;
          else if (m[i] == m[j]) e++;
        }
      }
      size_t o = (size_t)c * N + n;
      if (u2) u2[o] = 2 * g + e;
      if (gt) gt[o] = g;
      if (eq) eq[o] = e;
      if (pairs) pairs[o] = nm * nb;
      if (nm * nb > 0) {
        n_valid++;
        total_u2 += 2 * g + e;
        if (common < 0) common = nm * nb;
        else if (common != nm * nb) uniform = 0;
      }
    }
    double A;
    if (n_valid == 0) {
      A = NAN;
    } else if (uniform) {
      A = (double)total_u2 / (double)(2 * common * n_valid);
    } else {
      double acc = 0.0;
      for (uint32_t n = 0; n < N; ++n) {
        size_t o = (size_t)c * N + n;
        const int8_t *l = labels + o * S;
        int64_t nm = 0, nb = 0, g = 0, e = 0;
        const float *m = scores + o * S;
        for (uint32_t i = 0; i < S; ++i) {
          if (l[i] == 1) nm++;
          if (l[i] == 0) nb++;
        }
        if (nm * nb == 0) continue;
        for (uint32_t i = 0; i < S; ++i) {
          if (l[i] != 1) continue;
          for (uint32_t j = 0; j < S; ++j) {
            if (l[j] != 0) continue;
            if (m[i] > m[j]) g++;
            else if (m[i] == m[j]) e++;
          }
        }
        acc += (double)(2 * g + e) / (double)(2 * nm * nb);
      }
      A = acc / (double)n_valid;
    }
    if (auroc) auroc[c] = A;
  }
  return status;
}

/* Pooled Mann-Whitney AUROC: all malicious scores of a configuration      */
/* (every canary) against all its benign scores -- the U statistic the     */
/* paper names as equivalent to its ranking test (Sec. 3.4).  Brute force   */
/* over every (malicious, benign) pair of the configuration:               */
/*   u2 = 2 #{m_i > m_j} + #{m_i = m_j},  A = u2 / (2 n_mal n_ben).          */
/* NaN scores are left out of the pool and reported.                       */
int or_auroc_pooled(const float *scores, const int8_t *labels, uint32_t C,
                    uint32_t N, uint32_t S, int64_t *u2, int64_t *n_mal,
                    int64_t *n_ben, double *auroc) {
  int status = OR_OK;
  const size_t per = (size_t)N * S;
  for (uint32_t c = 0; c < C; ++c) {
    const float *m = scores + (size_t)c * per;
    const int8_t *l = labels + (size_t)c * per;
    int64_t g = 0, e = 0, nm = 0, nb = 0;
    for (size_t i = 0; i < per; ++i) {
      if ((l[i] == 1 || l[i] == 0) && isnan(m[i])) { status = OR_NAN_SCORE; continue; }
      if (l[i] == 1) nm++;
      if (l[i] == 0) nb++;
    }
    for (size_t i = 0; i < per; ++i) {
      if (l[i] != 1 || isnan(m[i])) continue;
      for (size_t j = 0; j < per; ++j) {
        if (l[j] != 0 || isnan(m[j])) continue;
        if (m[i] > m[j]) g++;
        else if (m[i] == m[j]) e++;
      }
    }
    if (u2) u2[c] = 2 * g + e;
    if (n_mal) n_mal[c] = nm;
    if (n_ben) n_ben[c] = nb;
    if (auroc)
      auroc[c] = (nm * nb > 0) ? (double)(2 * g + e) / (double)(2 * nm * nb) : NAN;
  }
  return status;
}

/* ------------------------------------------------------------------------ */
/* Scrambled-label negative control (Sec. 4.5): the true mismatches are kept */
/* and, on every canary, a stage j* drawn uniformly from the benign stages   */
/* takes the malicious label.  The truly malicious stages are left out       */
/* (label -1) so the remaining stages are exchangeable and E[A-hat] = 0.5.   */
/* labels/ctrl: [C][N][S]; the draw for (config c, canary n) uses aux        */
/* stream (purpose CONTROL, sub n) with counter word c2 = config_id0 + c.    */
int or_control_labels(const int8_t *labels, uint32_t C, uint32_t N,
                      uint32_t S, uint64_t seed, uint32_t config_id0,
                      int8_t *ctrl) {
  uint32_t *benign = (uint32_t *)malloc(S * sizeof(uint32_t));
  if (!benign) return OR_NO_MEMORY;
  int st = OR_OK;
  for (uint32_t c = 0; c < C; ++c) {
    for (uint32_t n = 0; n < N; ++n) {
      size_t o = ((size_t)c * N + n) * S;
      uint32_t b = 0;
      for (uint32_t s = 0; s < S; ++s)
        if (labels[o + s] == 0) benign[b++] = s;
      for (uint32_t s = 0; s < S; ++s)
        ctrl[o + s] = (labels[o + s] == 0) ? 0 : -1;
      if (b == 0) { st = OR_BAD_ARG; continue; }
      or_words w;
      words_init(&w, seed, OR_AUX_CONTROL, n, config_id0 + c);
      uint32_t r = words_bounded(&w, b);
      ctrl[o + benign[r]] = 1;
    }
  }
  free(benign);
  return st;
}

int or_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}
