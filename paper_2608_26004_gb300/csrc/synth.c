/*
 * Seeded synthetic inputs for the fuse-and-verify step.
 *
 * This file simulates the three forward passes that precede the step (the
 * drafter on the full context, the drafter on the compressed context and the
 * verifier on the compressed context, Section 3.2 of the paper) with random
 * logits, and the drafter's own sampling of the K draft tokens (Algorithm 1,
 * the drafting step).  It contains none of the step's arithmetic: no delta
 * fusion, no divergence, no gate, no acceptance test, no residual.
 *
 * Randomness is counter based, so every element has its own address and the
 * output does not depend on the thread count:
 *   Philox4x32-10 (Salmon, Moraes, Dror and Shaw, "Parallel Random Numbers:
 *   As Easy as 1, 2, 3", SC'11): 10 rounds of two 32x32->64 multiplies, with
 *   a Weyl-sequence key schedule.
 * Normals come from the Box-Muller transform.  The logarithm, sine, cosine and
 * exponential used here are written out below as plain series in IEEE double
 * arithmetic (compiled with -ffp-contract=off), so that x86-64 and aarch64
 * hosts produce bit-identical inputs.
 *
 * Layout of every logit tensor: [B, K+1, V] row-major, fp32 or bf16 (bf16 is
 * stored as raw uint16 bit patterns, rounded to nearest even from fp32).
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ---------------------------------------------------------------- Philox */

#define PHILOX_MUL0 0xD2511F53u
#define PHILOX_MUL1 0xCD9E8D57u
#define PHILOX_WEYL0 0x9E3779B9u
#define PHILOX_WEYL1 0xBB67AE85u

void asymspec_philox4x32_10(const uint32_t ctr_in[4], const uint32_t key_in[2],
                            uint32_t out[4]) {
  uint32_t c0 = ctr_in[0], c1 = ctr_in[1], c2 = ctr_in[2], c3 = ctr_in[3];
  uint32_t k0 = key_in[0], k1 = key_in[1];
  for (int round = 0; round < 10; ++round) {
    uint64_t p0 = (uint64_t)PHILOX_MUL0 * (uint64_t)c0;
    uint64_t p1 = (uint64_t)PHILOX_MUL1 * (uint64_t)c2;
    uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
    uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
    uint32_t n0 = hi1 ^ c1 ^ k0;
    uint32_t n2 = hi0 ^ c3 ^ k1;
    c0 = n0;
    c1 = lo1;
    c2 = n2;
    c3 = lo0;
    k0 += PHILOX_WEYL0;
    k1 += PHILOX_WEYL1;
  }
  out[0] = c0;
  out[1] = c1;
  out[2] = c2;
  out[3] = c3;
}

/* ------------------------------------------- deterministic elementary math */

static const double kLn2 = 0.6931471805599453094;
static const double kHalfPi = 1.5707963267948966192;

/* ln(x) for x > 0: x = m * 2^e with m in [sqrt(1/2), sqrt(2)), then
 * ln(m) = 2 atanh(z) = 2 (z + z^3/3 + z^5/5 + ...), z = (m-1)/(m+1). */
static double det_log(double x) {
  int e;
  double m = frexp(x, &e); /* m in [0.5, 1) */
  if (m < 0.70710678118654752440) {
    m *= 2.0;
    e -= 1;
  }
  double z = (m - 1.0) / (m + 1.0);
  double z2 = z * z;
  double term = z, sum = 0.0;
  for (int n = 1; n <= 27; n += 2) {
    sum = sum + term / (double)n;
    term = term * z2;
  }
  return 2.0 * sum + (double)e * kLn2;
}

/* exp(x) = 2^k e^r, k = nearest integer to x/ln2, e^r by its Taylor series. */
static double det_exp(double x) {
  if (x < -745.0) return 0.0;
  double kd = floor(x / kLn2 + 0.5);
  double r = x - kd * kLn2;
  double term = 1.0, sum = 1.0;
  for (int n = 1; n <= 18; ++n) {
    term = term * r / (double)n;
    sum = sum + term;
  }
  return ldexp(sum, (int)kd);
}

/* sin and cos of theta in [0, pi/2) by their Taylor series. */
static void det_sincos_quarter(double th, double* s, double* c) {
  double th2 = th * th;
  double ts = th, tc = 1.0, ss = 0.0, cc = 0.0;
  for (int n = 0; n < 14; ++n) {
    ss = ss + ts;
    cc = cc + tc;
    ts = -ts * th2 / (double)((2 * n + 2) * (2 * n + 3));
    tc = -tc * th2 / (double)((2 * n + 1) * (2 * n + 2));
  }
  *s = ss;
  *c = cc;
}

/* cos(2 pi u), sin(2 pi u) for u in [0, 1). */
static void det_sincos_turn(double u, double* s, double* c) {
  double q4 = u * 4.0; /* exact */
  double qf = floor(q4);
  int q = (int)qf & 3;
  double th = (q4 - qf) * kHalfPi;
  double s0, c0;
  det_sincos_quarter(th, &s0, &c0);
  switch (q) {
    case 0: *c = c0; *s = s0; break;
    case 1: *c = -s0; *s = c0; break;
    case 2: *c = -c0; *s = -s0; break;
    default: *c = s0; *s = -c0; break;
  }
}

/* ------------------------------------------------------------ primitives */

enum {
  TAG_VERIFIER = 1,  /* z_v noise */
  TAG_FULL = 2,      /* z_f noise */
  TAG_SELECT = 3,    /* which tokens of z_c are perturbed */
  TAG_PERTURB = 4,   /* z_c perturbation normals */
  TAG_ROW = 5,       /* per-row scalars */
  TAG_SHUFFLE = 6,   /* Fisher-Yates draws */
  TAG_PROFILE = 7    /* noise on the sorted Zipf profile */
};

typedef struct {
  uint32_t key[2];
} synth_key;

static void draw4(const synth_key* k, uint32_t tag, uint32_t b, uint32_t kk,
                  uint32_t j, uint32_t out[4]) {
  uint32_t ctr[4] = {tag, b, kk, j};
  asymspec_philox4x32_10(ctr, k->key, out);
}

/* 32-bit word -> U(0,1) excluding 0 (used as the Box-Muller radius input). */
static double u_open(uint32_t w) { return ((double)w + 0.5) * (1.0 / 4294967296.0); }
/* 32-bit word -> U[0,1). */
static double u_half(uint32_t w) { return (double)w * (1.0 / 4294967296.0); }
/* 32-bit word -> U[0,1) with 24 bits (exactly representable in fp32). */
static double u_24(uint32_t w) { return (double)(w >> 8) * (1.0 / 16777216.0); }

/* Four standard normals for elements 4j..4j+3 of stream (tag, b, k). */
static void normals4(const synth_key* k, uint32_t tag, uint32_t b, uint32_t kk,
                     uint32_t j, double out[4]) {
  uint32_t w[4];
  draw4(k, tag, b, kk, j, w);
  for (int h = 0; h < 2; ++h) {
    double r = sqrt(-2.0 * det_log(u_open(w[2 * h])));
    double s, c;
    det_sincos_turn(u_half(w[2 * h + 1]), &s, &c);
    out[2 * h] = r * c;
    out[2 * h + 1] = r * s;
  }
}

static uint16_t f32_to_bf16_rne(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  uint32_t bias = 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)((u + bias) >> 16);
}

static float bf16_to_f32(uint16_t h) {
  uint32_t u = (uint32_t)h << 16;
  float f;
  memcpy(&f, &u, 4);
  return f;
}

/* ---------------------------------------------------------------- recipe */

typedef struct {
  int profile;          /* 0: N(0, sigma_v^2) + spike; 1: sorted Zipf + noise, permuted */
  double sigma_v;       /* profile 0 */
  double spike;         /* profile 0: added to one uniformly drawn token per row */
  double zipf_s;        /* profile 1: value at rank r is -zipf_s * ln r */
  double zipf_noise;    /* profile 1: N(0, zipf_noise^2) added per rank */
  double sigma_f;       /* z_f = z_v + N(0, sigma_f^2) */
  double frac_lo;       /* fraction of tokens of z_c perturbed, drawn per row */
  double frac_hi;       /*   uniformly from [frac_lo, frac_hi] */
  double sigma_c;       /* perturbation N(0, sigma_c^2) */
  int identical_lower_half; /* rows with b < B_total/2 keep z_c == z_f */
} asymspec_recipe;

typedef struct {
  const asymspec_recipe* rc;
  synth_key key;
  int b0, nb, B_total, K, V, dtype;
  void *full, *comp, *ver;
  int32_t* tokens;
  float* probs;
  float* unif;
  int next_row; /* shared work counter, guarded by mu */
  pthread_mutex_t mu;
} synth_job;

static void store(void* base, int dtype, size_t idx, double x, float* stored) {
  float f = (float)x;
  if (dtype == 0) {
    ((float*)base)[idx] = f;
    *stored = f;
  } else {
    uint16_t h = f32_to_bf16_rne(f);
    ((uint16_t*)base)[idx] = h;
    *stored = bf16_to_f32(h);
  }
}

static void make_row(synth_job* job, int bl, int k, double* zv, double* zf,
                     double* zc, float* fstore, uint32_t* perm, double* work) {
  const asymspec_recipe* rc = job->rc;
  const int V = job->V, K = job->K;
  const uint32_t b = (uint32_t)(job->b0 + bl);
  uint32_t rw[4];
  draw4(&job->key, TAG_ROW, b, (uint32_t)k, 0, rw);
  double nrm[4];

  /* verifier logits z_v */
  if (rc->profile == 0) {
    for (int v = 0; v < V; v += 4) {
      normals4(&job->key, TAG_VERIFIER, b, (uint32_t)k, (uint32_t)(v >> 2), nrm);
      for (int e = 0; e < 4 && v + e < V; ++e) zv[v + e] = rc->sigma_v * nrm[e];
    }
    uint32_t spike_at = (uint32_t)(((uint64_t)rw[0] * (uint64_t)V) >> 32);
    zv[spike_at] += rc->spike;
  } else {
    for (int v = 0; v < V; ++v) perm[v] = (uint32_t)v;
    uint32_t sw[4];
    for (int i = V - 1; i >= 1; --i) {
      if (i == V - 1 || (i & 3) == 3)
        draw4(&job->key, TAG_SHUFFLE, b, (uint32_t)k, (uint32_t)(i >> 2), sw);
      uint32_t j = (uint32_t)(((uint64_t)sw[i & 3] * (uint64_t)(i + 1)) >> 32);
      uint32_t tmp = perm[i];
      perm[i] = perm[j];
      perm[j] = tmp;
    }
    for (int r = 0; r < V; r += 4) {
      normals4(&job->key, TAG_PROFILE, b, (uint32_t)k, (uint32_t)(r >> 2), nrm);
      for (int e = 0; e < 4 && r + e < V; ++e)
        zv[perm[r + e]] = -rc->zipf_s * det_log((double)(r + e + 1)) + rc->zipf_noise * nrm[e];
    }
  }

  /* drafter on the full context: z_f = z_v + noise */
  for (int v = 0; v < V; v += 4) {
    normals4(&job->key, TAG_FULL, b, (uint32_t)k, (uint32_t)(v >> 2), nrm);
    for (int e = 0; e < 4 && v + e < V; ++e) zf[v + e] = zv[v + e] + rc->sigma_f * nrm[e];
  }

  /* drafter on the compressed context: z_f with a fraction of tokens shifted */
  int identical = rc->identical_lower_half && ((int)b < job->B_total / 2);
  double frac = rc->frac_lo + (rc->frac_hi - rc->frac_lo) * u_24(rw[1]);
  for (int v = 0; v < V; v += 4) {
    uint32_t sel[4];
    draw4(&job->key, TAG_SELECT, b, (uint32_t)k, (uint32_t)(v >> 2), sel);
    normals4(&job->key, TAG_PERTURB, b, (uint32_t)k, (uint32_t)(v >> 2), nrm);
    for (int e = 0; e < 4 && v + e < V; ++e) {
      double x = zf[v + e];
      if (!identical && u_24(sel[e]) < frac) x += rc->sigma_c * nrm[e];
      zc[v + e] = x;
    }
  }

  size_t row = ((size_t)bl * (size_t)(K + 1) + (size_t)k) * (size_t)V;
  for (int v = 0; v < V; ++v) {
    float tmp;
    store(job->ver, job->dtype, row + v, zv[v], &tmp);
    store(job->full, job->dtype, row + v, zf[v], &fstore[v]);
    store(job->comp, job->dtype, row + v, zc[v], &tmp);
  }

  /* the drafter samples d_{k+1} from softmax of its stored full-context logits */
  if (k < K) {
    double mx = -INFINITY;
    for (int v = 0; v < V; ++v)
      if ((double)fstore[v] > mx) mx = (double)fstore[v];
    double tot = 0.0;
    for (int v = 0; v < V; ++v) {
      work[v] = det_exp((double)fstore[v] - mx);
      tot += work[v];
    }
    double u = u_24(rw[2]);
    double cum = 0.0;
    int pick = -1, last_pos = 0;
    for (int v = 0; v < V; ++v) {
      double p = work[v] / tot;
      if (p > 0.0) last_pos = v;
      cum += p;
      if (cum > u) {
        pick = v;
        break;
      }
    }
    if (pick < 0) pick = last_pos;
    job->tokens[(size_t)bl * K + k] = pick;
    job->probs[(size_t)bl * K + k] = (float)(work[pick] / tot);
  }
  job->unif[(size_t)bl * (K + 1) + k] = (float)u_24(rw[3]);
}

static void* synth_worker(void* arg) {
  synth_job* job = (synth_job*)arg;
  const int V = job->V;
  double* zv = (double*)malloc(sizeof(double) * (size_t)V * 4);
  float* fstore = (float*)malloc(sizeof(float) * (size_t)V);
  uint32_t* perm = (uint32_t*)malloc(sizeof(uint32_t) * (size_t)V);
  if (!zv || !fstore || !perm) {
    free(zv);
    free(fstore);
    free(perm);
    return (void*)1;
  }
  double *zf = zv + V, *zc = zv + 2 * (size_t)V, *work = zv + 3 * (size_t)V;
  const int rows = job->nb * (job->K + 1);
  for (;;) {
    pthread_mutex_lock(&job->mu);
    int r = job->next_row++;
    pthread_mutex_unlock(&job->mu);
    if (r >= rows) break;
    make_row(job, r / (job->K + 1), r % (job->K + 1), zv, zf, zc, fstore, perm, work);
  }
  free(zv);
  free(fstore);
  free(perm);
  return NULL;
}

/*
 * Fills batch elements [b0, b0+nb) of a configuration whose full batch is
 * B_total.  Rows of a batch element are identical whatever b0/nb are, so a
 * sample of a large configuration can be generated on its own.
 * Host buffers: full/comp/ver [nb, K+1, V] (dtype 0 = fp32, 1 = bf16 bits),
 * tokens/probs [nb, K], unif [nb, K+1].  Returns 0 on success.
 */
int asymspec_synth_generate(const asymspec_recipe* rc, uint64_t seed, int b0, int nb,
                            int B_total, int K, int V, int dtype, void* full,
                            void* comp, void* ver, int32_t* tokens, float* probs,
                            float* unif, int nthreads) {
  if (!rc || nb < 0 || b0 < 0 || K < 1 || V < 2 || (dtype != 0 && dtype != 1)) return -1;
  if (nb == 0) return 0;
  if (!full || !comp || !ver || !tokens || !probs || !unif) return -1;
  synth_job job;
  job.rc = rc;
  job.key.key[0] = (uint32_t)seed;
  job.key.key[1] = (uint32_t)(seed >> 32);
  job.b0 = b0;
  job.nb = nb;
  job.B_total = B_total;
  job.K = K;
  job.V = V;
  job.dtype = dtype;
  job.full = full;
  job.comp = comp;
  job.ver = ver;
  job.tokens = tokens;
  job.probs = probs;
  job.unif = unif;
  job.next_row = 0;
  pthread_mutex_init(&job.mu, NULL);
  if (nthreads < 1) nthreads = 1;
  if (nthreads > 64) nthreads = 64;
  pthread_t th[64];
  int started = 0, rc_all = 0;
  for (int i = 1; i < nthreads; ++i) {
    if (pthread_create(&th[started], NULL, synth_worker, &job) == 0) ++started;
  }
  if (synth_worker(&job) != NULL) rc_all = -2;
  for (int i = 0; i < started; ++i) {
    void* ret = NULL;
    pthread_join(th[i], &ret);
    if (ret != NULL) rc_all = -2;
  }
  pthread_mutex_destroy(&job.mu);
  return rc_all;
}
