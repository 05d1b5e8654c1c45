/*
 * ntc_oracle.c -- plain, slow CPU oracle for the runtime decode of
 * neural-compressed textures ("Thread-Efficient Decoding for Neural Texture
 * Compression", Sec. 2 and Sec. 3.3).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may link or call this
 * file; only the test suite, the smoke check and the benchmark's CPU-baseline
 * leg do.  It shares no code, header, table or helper with the CUDA library.
 *
 * What it computes, per query q = (set id s, u, v, lod):
 *   Sec. 3.3: the texel is x^ = D_{c(s)}(z_s): the latents z_s of texture set s
 *   are decoded by the decoder assigned to the set's cluster c(s).
 *   Sec. 4 (experimental setup): the decoder is a 3-layer MLP whose first two
 *   layers are hidden layers; the latents form a grid ("latent pyramids or
 *   grids", Sec. 1).
 * The paper does not spell out the sampling rule, mip handling or the MLP I/O,
 * so this file implements the following reading, step by step:
 *   1. dec = map[s]; a set id >= num_sets, or a non-finite u or v, makes the
 *      query "bad": every output channel is NaN.
 *   2. lambda = fmaxf(lod, 0); lo = min(floor(lambda), num_mips-1);
 *      t = (lo == num_mips-1) ? 0 : lambda - lo                     (fp32)
 *   3. For every latent level k and every used mip m (lo, and lo+1 when t>0),
 *      with W, H = max(1, W0>>m), max(1, H0>>m), in fp32 round-to-nearest with
 *      no contraction (this file is compiled with -ffp-contract=off):
 *        wrap : uw = u - floorf(u), x = uw*W - 0.5
 *        clamp: x = u*W - 0.5
 *        x0 = floorf(x), wx = x - x0   (same for y)
 *        wrap : i0 = x0 mod W, i1 = (x0+1) mod W     (non-negative modulo)
 *        clamp: i0 = clamp(x0, 0, W-1), i1 = clamp(x0+1, 0, W-1)
 *        weights w00=(1-wx)(1-wy), w10=wx(1-wy), w01=(1-wx)wy, w11=wx*wy
 *        tap order (i0,j0), (i1,j0), (i0,j1), (i1,j1)
 *        texel index = base(s,k,m) + j*W + i
 *   4. f_k[c] = sum_taps w * L[tap][c] in double; with t > 0 the level feature
 *      is (1-t) f_k(lo) + t f_k(lo+1).  f = [f_0 | f_1 | ... | pe].
 *      Positional encoding (Sec. 4: the encoder output "is concatenated with
 *      positional encoding"; its form is not given), F frequencies: with u', v'
 *      the coordinates the taps use (wrapped into [0,1) in wrap mode, as given
 *      in clamp mode, fp32), pe[4k..4k+3] = sin(2 pi 2^k u'), cos(2 pi 2^k u'),
 *      sin(2 pi 2^k v'), cos(2 pi 2^k v') for k < F, in double.
 *   5. MLP in double: h = act(W1 f + b1); h = act(Wl h + bl) for each further
 *      hidden layer; o = 1 / (1 + exp(-(Wout h + bout))).  act is ReLU, or
 *      LeakyReLU (Sec. 4) x > 0 ? x : slope * x.  Weights are stored per
 *      decoder as W1[H][IN], b1[H], {W[H][H], b[H]}..., Wout[C][H], bout[C].
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* Query record, 16 bytes: set id, u, v, lod. */
typedef struct {
  uint32_t set_id;
  float u, v, lod;
} or_query;

/* Everything the decode reads.  Arrays are host memory owned by the caller. */
typedef struct {
  uint32_t num_sets;
  uint32_t num_levels;    /* latent levels concatenated into the MLP input   */
  uint32_t num_mips;      /* mip-chain length of every level                  */
  uint32_t channels;      /* channels per latent texel                        */
  const uint32_t *level_dims;     /* [num_sets][num_levels][2]: W, H of mip 0 */
  const uint64_t *latent_offsets; /* [num_sets][num_levels][num_mips], texels */
  const uint16_t *latents;        /* IEEE half bits, [texel][channel]         */
  uint32_t address_mode;          /* 0 = wrap, 1 = clamp                      */
  uint32_t num_decoders;
  uint32_t in_dim, hidden, num_hidden_layers, out_dim;
  const float *weights;           /* [num_decoders][params per decoder]       */
  const uint32_t *set_to_decoder; /* [num_sets]                               */
  uint32_t pe_frequencies;        /* F: 4F positional-encoding inputs         */
  uint32_t activation;            /* 0 = ReLU, 1 = LeakyReLU                  */
  float leaky_slope;              /* LeakyReLU slope for x <= 0               */
} or_assets;

/* IEEE-754 binary16 -> double, written from the format's definition
 * (1 sign bit, 5 exponent bits with bias 15, 10 fraction bits). */
static double or_half_to_double(uint16_t h) {
  int sign = (h >> 15) & 1;
  int e = (h >> 10) & 0x1f;
  int f = h & 0x3ff;
  double v;
  if (e == 0)
    v = ldexp((double)f, -24); /* subnormal: f * 2^-14 * 2^-10 */
  else if (e == 31)
    v = f ? NAN : INFINITY;
  else
    v = ldexp((double)(1024 + f), e - 25); /* (1 + f/1024) * 2^(e-15) */
  return sign ? -v : v;
}

static size_t or_params_per_decoder(const or_assets *a) {
  size_t H = a->hidden, I = a->in_dim, C = a->out_dim;
  return H * I + H + (size_t)(a->num_hidden_layers - 1) * (H * H + H) + C * H + C;
}

/* Step 2: mip selection.  Returns lo, writes the blend factor t. */
static int or_select_mip(const or_assets *a, float lod, float *t_out) {
  float lam = fmaxf(lod, 0.0f);
  float lof = fminf(floorf(lam), (float)(a->num_mips - 1));
  int lo = (int)lof;
  float t = (lo == (int)a->num_mips - 1) ? 0.0f : lam - lof;
  *t_out = t;
  return lo;
}

/* Step 3 along one axis: texel indices and the fractional weight. */
static void or_axis(float c, uint32_t n, uint32_t mode, int64_t *i0, int64_t *i1,
                    float *frac) {
  float x;
  if (mode == 0) {
    float cw = c - floorf(c);
    x = cw * (float)n - 0.5f;
  } else {
    x = c * (float)n - 0.5f;
  }
  float x0f = floorf(x);
  *frac = x - x0f;
  if (mode == 0) {
    int64_t x0 = (int64_t)x0f; /* in [-1, n-1] because cw is in [0, 1] */
    int64_t a0 = x0 % (int64_t)n, a1 = (x0 + 1) % (int64_t)n;
    if (a0 < 0) a0 += n;
    if (a1 < 0) a1 += n;
    *i0 = a0;
    *i1 = a1;
  } else {
    float xc = fminf(fmaxf(x0f, -1.0f), (float)n);
    int64_t x0 = (int64_t)xc;
    int64_t a0 = x0, a1 = x0 + 1;
    if (a0 < 0) a0 = 0;
    if (a0 > (int64_t)n - 1) a0 = (int64_t)n - 1;
    if (a1 < 0) a1 = 0;
    if (a1 > (int64_t)n - 1) a1 = (int64_t)n - 1;
    *i0 = a0;
    *i1 = a1;
  }
}

/* Step 3 for one (set, level, mip): 4 texel indices and 4 fp32 weights. */
static void or_bilinear_taps(const or_assets *a, uint32_t s, uint32_t k, uint32_t m,
                             float u, float v, uint64_t idx[4], float w[4]) {
  uint32_t W0 = a->level_dims[((size_t)s * a->num_levels + k) * 2 + 0];
  uint32_t H0 = a->level_dims[((size_t)s * a->num_levels + k) * 2 + 1];
  uint32_t W = W0 >> m, H = H0 >> m;
  if (W < 1) W = 1;
  if (H < 1) H = 1;
  uint64_t base = a->latent_offsets[((size_t)s * a->num_levels + k) * a->num_mips + m];
  int64_t i0, i1, j0, j1;
  float wx, wy;
  or_axis(u, W, a->address_mode, &i0, &i1, &wx);
  or_axis(v, H, a->address_mode, &j0, &j1, &wy);
  idx[0] = base + (uint64_t)j0 * W + (uint64_t)i0;
  idx[1] = base + (uint64_t)j0 * W + (uint64_t)i1;
  idx[2] = base + (uint64_t)j1 * W + (uint64_t)i0;
  idx[3] = base + (uint64_t)j1 * W + (uint64_t)i1;
  float ax = 1.0f - wx, ay = 1.0f - wy;
  w[0] = ax * ay;
  w[1] = wx * ay;
  w[2] = ax * wy;
  w[3] = wx * wy;
}

static int or_query_is_bad(const or_assets *a, const or_query *q) {
  return q->set_id >= a->num_sets || !isfinite(q->u) || !isfinite(q->v);
}

/* Steps 1-4 for one query: the MLP input vector f (length in_dim =
 * num_levels*channels + 4*pe_frequencies).  Returns 0 for a bad query (f
 * untouched). */
static int or_features_one(const or_assets *a, const or_query *q, double *f) {
  if (or_query_is_bad(a, q)) return 0;
  float t;
  int lo = or_select_mip(a, q->lod, &t);
  const uint32_t C = a->channels;
  for (uint32_t k = 0; k < a->num_levels; ++k) {
    int nm = (t > 0.0f) ? 2 : 1;
    double acc[2][64];
    for (int mi = 0; mi < nm; ++mi) {
      uint64_t idx[4];
      float w[4];
      or_bilinear_taps(a, q->set_id, k, (uint32_t)(lo + mi), q->u, q->v, idx, w);
      for (uint32_t c = 0; c < C; ++c) {
        double sum = 0.0;
        for (int tp = 0; tp < 4; ++tp)
          sum += (double)w[tp] * or_half_to_double(a->latents[idx[tp] * C + c]);
        acc[mi][c] = sum;
      }
    }
    for (uint32_t c = 0; c < C; ++c)
      f[k * C + c] = (nm == 2) ? (1.0 - (double)t) * acc[0][c] + (double)t * acc[1][c]
                               : acc[0][c];
  }
  const double two_pi = 6.283185307179586476925286766559;
  const float uw = a->address_mode == 0 ? q->u - floorf(q->u) : q->u;
  const float vw = a->address_mode == 0 ? q->v - floorf(q->v) : q->v;
  double *pe = f + (size_t)a->num_levels * C;
  for (uint32_t k = 0; k < a->pe_frequencies; ++k) {
    const double su = two_pi * ldexp((double)uw, (int)k), sv = two_pi * ldexp((double)vw, (int)k);
    pe[4 * k + 0] = sin(su);
    pe[4 * k + 1] = cos(su);
    pe[4 * k + 2] = sin(sv);
    pe[4 * k + 3] = cos(sv);
  }
  return 1;
}

static double or_act(const or_assets *a, double x) {
  if (x > 0.0) return x;
  return a->activation == 1 ? (double)a->leaky_slope * x : 0.0;
}

/* Step 5: the decoder MLP in double. */
static void or_mlp(const or_assets *a, uint32_t dec, const double *f, double *o) {
  const uint32_t I = a->in_dim, H = a->hidden, C = a->out_dim;
  const float *p = a->weights + (size_t)dec * or_params_per_decoder(a);
  double *h = (double *)malloc(sizeof(double) * H);
  double *g = (double *)malloc(sizeof(double) * H);
  /* layer 1 */
  const float *W = p, *b = p + (size_t)H * I;
  for (uint32_t j = 0; j < H; ++j) {
    double acc = (double)b[j];
    for (uint32_t i = 0; i < I; ++i) acc += (double)W[(size_t)j * I + i] * f[i];
    h[j] = or_act(a, acc);
  }
  p = b + H;
  /* further hidden layers */
  for (uint32_t l = 1; l < a->num_hidden_layers; ++l) {
    W = p;
    b = p + (size_t)H * H;
    for (uint32_t j = 0; j < H; ++j) {
      double acc = (double)b[j];
      for (uint32_t i = 0; i < H; ++i) acc += (double)W[(size_t)j * H + i] * h[i];
      g[j] = or_act(a, acc);
    }
    memcpy(h, g, sizeof(double) * H);
    p = b + H;
  }
  /* output layer + sigmoid */
  W = p;
  b = p + (size_t)C * H;
  for (uint32_t c = 0; c < C; ++c) {
    double acc = (double)b[c];
    for (uint32_t i = 0; i < H; ++i) acc += (double)W[(size_t)c * H + i] * h[i];
    o[c] = 1.0 / (1.0 + exp(-acc));
  }
  free(h);
  free(g);
}

/* ---------------------------------------------------------------- exports */

size_t or_param_count(const or_assets *a) { return or_params_per_decoder(a); }

/* Taps of every query: idx[n][num_levels][2][4], w[n][num_levels][2][4], t[n].
 * The second mip slot is filled only when t > 0; otherwise (and for a bad
 * query, everywhere) idx = UINT64_MAX and w = 0. */
void or_taps(const or_assets *a, const or_query *q, size_t n, uint64_t *idx, float *w,
             float *t_out) {
  const size_t per = (size_t)a->num_levels * 8;
  for (size_t i = 0; i < n; ++i) {
    uint64_t *I = idx + i * per;
    float *Wt = w + i * per;
    for (size_t e = 0; e < per; ++e) {
      I[e] = UINT64_MAX;
      Wt[e] = 0.0f;
    }
    t_out[i] = 0.0f;
    if (or_query_is_bad(a, &q[i])) continue;
    float t;
    int lo = or_select_mip(a, q[i].lod, &t);
    t_out[i] = t;
    for (uint32_t k = 0; k < a->num_levels; ++k) {
      or_bilinear_taps(a, q[i].set_id, k, (uint32_t)lo, q[i].u, q[i].v, I + k * 8,
                       Wt + k * 8);
      if (t > 0.0f)
        or_bilinear_taps(a, q[i].set_id, k, (uint32_t)lo + 1, q[i].u, q[i].v,
                         I + k * 8 + 4, Wt + k * 8 + 4);
    }
  }
}

/* MLP inputs of every query, f[n][in_dim]; NaN rows for bad ones. */
void or_features(const or_assets *a, const or_query *q, size_t n, double *f) {
  const size_t F = a->in_dim;
  for (size_t i = 0; i < n; ++i)
    if (!or_features_one(a, &q[i], f + i * F))
      for (size_t c = 0; c < F; ++c) f[i * F + c] = NAN;
}

/* Decode queries [begin, end): out[i][out_dim]. */
static void or_decode_range(const or_assets *a, const or_query *q, size_t begin,
                            size_t end, double *out) {
  const size_t F = a->in_dim;
  double *f = (double *)malloc(sizeof(double) * F);
  for (size_t i = begin; i < end; ++i) {
    double *o = out + i * a->out_dim;
    if (!or_features_one(a, &q[i], f)) {
      for (uint32_t c = 0; c < a->out_dim; ++c) o[c] = NAN;
      continue;
    }
    or_mlp(a, a->set_to_decoder[q[i].set_id], f, o);
  }
  free(f);
}

typedef struct {
  const or_assets *a;
  const or_query *q;
  size_t begin, end;
  double *out;
} or_job;

static void *or_worker(void *p) {
  or_job *j = (or_job *)p;
  or_decode_range(j->a, j->q, j->begin, j->end, j->out);
  return NULL;
}

/* Decode all n queries on nthreads host threads, each over a contiguous range.
 * Returns the number of bad queries. */
uint64_t or_decode(const or_assets *a, const or_query *q, size_t n, double *out,
                   int nthreads) {
  if (nthreads < 1) nthreads = 1;
  if ((size_t)nthreads > n) nthreads = n ? (int)n : 1;
  pthread_t *th = (pthread_t *)malloc(sizeof(pthread_t) * nthreads);
  or_job *jobs = (or_job *)malloc(sizeof(or_job) * nthreads);
  for (int t = 0; t < nthreads; ++t) {
    jobs[t].a = a;
    jobs[t].q = q;
    jobs[t].begin = n * (size_t)t / nthreads;
    jobs[t].end = n * (size_t)(t + 1) / nthreads;
    jobs[t].out = out;
    if (t > 0) pthread_create(&th[t], NULL, or_worker, &jobs[t]);
  }
  or_worker(&jobs[0]);
  for (int t = 1; t < nthreads; ++t) pthread_join(th[t], NULL);
  free(th);
  free(jobs);
  uint64_t bad = 0;
  for (size_t i = 0; i < n; ++i) bad += (uint64_t)or_query_is_bad(a, &q[i]);
  return bad;
}

/* ------------------------------------------------------------------ k-means
 * Alg. 2, Stage 2 ("Clustering into m groups", Sec. 3.3): k-means over the
 * per-texture embeddings F [n][dim] into m groups gives the assignment c(i),
 * i.e. the set -> decoder map.  The paper names k-means and nothing else; this
 * is Lloyd's iteration with the following reading:
 *   start       mu_g = F[init[g]] for g < m (the caller picks m distinct sets)
 *   assignment  c(i) = argmin_g sum_j (F[i][j] - mu_g[j])^2, in double, the sum
 *               taken over j in increasing order; ties go to the smallest g
 *   update      mu_g = (sum of F[i] over c(i) = g, i increasing) / |group g|;
 *               an empty group keeps its centroid
 *   stop        when an assignment equals the previous one, or after max_iters
 *               assignments
 * Returns the number of assignments made; map[n] is the last assignment and
 * centroids[m][dim] the means of that assignment (the last update). */
uint32_t or_kmeans(const float *F, uint32_t n, uint32_t dim, uint32_t m, const uint32_t *init,
                   uint32_t max_iters, uint32_t *map, double *centroids) {
  double *mu = centroids;
  for (uint32_t g = 0; g < m; ++g)
    for (uint32_t j = 0; j < dim; ++j) mu[(size_t)g * dim + j] = (double)F[(size_t)init[g] * dim + j];
  for (uint32_t i = 0; i < n; ++i) map[i] = 0xFFFFFFFFu;
  uint32_t t = 0;
  while (t < max_iters) {
    ++t;
    int changed = 0;
    for (uint32_t i = 0; i < n; ++i) {
      uint32_t best = 0;
      double best_d = 0.0;
      for (uint32_t g = 0; g < m; ++g) {
        double dist = 0.0;
        for (uint32_t j = 0; j < dim; ++j) {
          const double d = (double)F[(size_t)i * dim + j] - mu[(size_t)g * dim + j];
          dist = dist + d * d;
        }
        if (g == 0 || dist < best_d) {
          best = g;
          best_d = dist;
        }
      }
      if (map[i] != best) changed = 1;
      map[i] = best;
    }
    if (!changed) break;
    for (uint32_t g = 0; g < m; ++g) {
      uint64_t count = 0;
      for (uint32_t i = 0; i < n; ++i) count += map[i] == g;
      if (count == 0) continue;
      for (uint32_t j = 0; j < dim; ++j) {
        double s = 0.0;
        for (uint32_t i = 0; i < n; ++i)
          if (map[i] == g) s = s + (double)F[(size_t)i * dim + j];
        mu[(size_t)g * dim + j] = s / (double)count;
      }
    }
  }
  return t;
}
