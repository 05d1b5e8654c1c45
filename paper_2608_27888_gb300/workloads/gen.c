/*
 * gen.c -- seeded synthetic inputs for the neural-texture decode: latent
 * pyramids with box-filtered mip chains, decoder weights, set->decoder maps and
 * query streams (uniform, texel-centre raster, Voronoi G-buffer, controlled
 * divergence per 32-query warp).
 *
 * This file holds input generation only, none of the decode's arithmetic; the
 * CUDA library and the CPU oracle both consume what it writes.  Every random
 * number comes from SplitMix64 (Steele, Lea and Flood, "Fast splittable
 * pseudorandom number generators", OOPSLA 2014) used as a counter-based
 * generator: draw i of a stream with key k is mix(k + (i + 1) * gamma).
 * Normals use the Box-Muller transform (Box and Muller, 1958) in double.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define GAMMA 0x9E3779B97F4A7C15ULL
#define TWO_PI 6.283185307179586476925286766559

static uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

uint64_t gen_key(uint64_t seed, uint64_t tag, uint64_t a, uint64_t b) {
  return mix64(mix64(mix64(seed ^ (tag * GAMMA)) + a * GAMMA) ^ (b + 0x632BE59BD9B4E019ULL));
}

static inline uint64_t draw(uint64_t key, uint64_t i) { return mix64(key + (i + 1) * GAMMA); }
/* uniform double in [0, 1) from the top 53 bits */
static inline double unif(uint64_t key, uint64_t i) {
  return (double)(draw(key, i) >> 11) * (1.0 / 9007199254740992.0);
}
/* uniform integer in [0, n) by multiply-shift of the top 32 bits */
static inline uint32_t unif_int(uint64_t key, uint64_t i, uint32_t n) {
  return (uint32_t)(((draw(key, i) >> 32) * (uint64_t)n) >> 32);
}

/* IEEE binary16 with round-to-nearest-even, from a double. */
uint16_t gen_double_to_half(double x) {
  uint16_t sign = signbit(x) ? 0x8000 : 0;
  double a = fabs(x);
  if (isnan(x)) return sign | 0x7e00;
  if (a >= 65520.0) return sign | 0x7c00;
  if (a < 6.103515625e-05) { /* below 2^-14: subnormal grid of 2^-24 */
    double r = rint(a * 16777216.0);
    return sign | (uint16_t)r; /* r == 1024 is the smallest normal */
  }
  int E;
  frexp(a, &E); /* a = f * 2^E, f in [0.5, 1) */
  int e = E - 1;
  uint32_t m = (uint32_t)rint(ldexp(a, 10 - e)); /* in [1024, 2048] */
  if (m == 2048) {
    m = 1024;
    e += 1;
  }
  if (e > 15) return sign | 0x7c00;
  return sign | (uint16_t)((e + 15) << 10) | (uint16_t)(m - 1024);
}

static float half_to_float_gen(uint16_t h) {
  int s = (h >> 15) & 1, e = (h >> 10) & 0x1f, f = h & 0x3ff;
  float v;
  if (e == 0) v = ldexpf((float)f, -24);
  else if (e == 31) v = f ? NAN : INFINITY;
  else v = ldexpf((float)(1024 + f), e - 25);
  return s ? -v : v;
}

/* Normals N(0, sigma) rounded to fp16: element i belongs to Box-Muller pair
 * i/2, whose two uniforms are draws 2*(i/2) and 2*(i/2)+1 of stream key. */
static void normals_f16(uint64_t key, uint64_t count, double sigma, uint16_t *out) {
  for (uint64_t p = 0; 2 * p < count; ++p) {
    double u1 = unif(key, 2 * p), u2 = unif(key, 2 * p + 1);
    double r = sqrt(-2.0 * log(1.0 - u1)) * sigma;
    out[2 * p] = gen_double_to_half(r * cos(TWO_PI * u2));
    if (2 * p + 1 < count) out[2 * p + 1] = gen_double_to_half(r * sin(TWO_PI * u2));
  }
}

/* One box-filter step of a mip chain: child texel (i, j) is the fp32 mean of the
 * parent's 2x2 block (indices clamped to the parent), rounded to fp16. */
static void mip_down(const uint16_t *p, uint32_t Wp, uint32_t Hp, uint32_t C, uint16_t *c,
                     uint32_t Wc, uint32_t Hc) {
  for (uint32_t j = 0; j < Hc; ++j)
    for (uint32_t i = 0; i < Wc; ++i) {
      uint32_t x0 = 2 * i < Wp ? 2 * i : Wp - 1, x1 = 2 * i + 1 < Wp ? 2 * i + 1 : Wp - 1;
      uint32_t y0 = 2 * j < Hp ? 2 * j : Hp - 1, y1 = 2 * j + 1 < Hp ? 2 * j + 1 : Hp - 1;
      for (uint32_t ch = 0; ch < C; ++ch) {
        float s = half_to_float_gen(p[((size_t)y0 * Wp + x0) * C + ch]);
        s = s + half_to_float_gen(p[((size_t)y0 * Wp + x1) * C + ch]);
        s = s + half_to_float_gen(p[((size_t)y1 * Wp + x0) * C + ch]);
        s = s + half_to_float_gen(p[((size_t)y1 * Wp + x1) * C + ch]);
        float m = s * 0.25f;
        c[((size_t)j * Wc + i) * C + ch] = gen_double_to_half((double)m);
      }
    }
}

typedef struct {
  uint64_t seed;
  uint32_t S, L, M, C;
  const uint32_t *dims;
  const uint64_t *offs;
  uint16_t *out;
  double sigma;
  uint32_t next; /* shared work counter over (set, level) pairs */
  pthread_mutex_t mu;
} lat_job;

static void *lat_worker(void *arg) {
  lat_job *J = (lat_job *)arg;
  for (;;) {
    pthread_mutex_lock(&J->mu);
    uint32_t w = J->next++;
    pthread_mutex_unlock(&J->mu);
    if (w >= J->S * J->L) break;
    uint32_t s = w / J->L, k = w % J->L;
    uint32_t W = J->dims[(size_t)w * 2], H = J->dims[(size_t)w * 2 + 1];
    uint16_t *base = J->out + J->offs[(size_t)w * J->M] * J->C;
    normals_f16(gen_key(J->seed, 1, s, k), (uint64_t)W * H * J->C, J->sigma, base);
    for (uint32_t m = 1; m < J->M; ++m) {
      uint32_t Wp = W >> (m - 1), Hp = H >> (m - 1), Wc = W >> m, Hc = H >> m;
      if (Wp < 1) Wp = 1;
      if (Hp < 1) Hp = 1;
      if (Wc < 1) Wc = 1;
      if (Hc < 1) Hc = 1;
      mip_down(J->out + J->offs[(size_t)w * J->M + m - 1] * J->C, Wp, Hp, J->C,
               J->out + J->offs[(size_t)w * J->M + m] * J->C, Wc, Hc);
    }
  }
  return NULL;
}

/* Latent pyramids: mip 0 of every (set, level) is N(0, sigma) in fp16, mips
 * 1..M-1 are its box-filtered chain.  dims[S][L][2], offs[S][L][M] (texels). */
void gen_latents(uint64_t seed, uint32_t S, uint32_t L, uint32_t M, uint32_t C,
                 const uint32_t *dims, const uint64_t *offs, double sigma, uint16_t *out,
                 int nthreads) {
  lat_job J = {.seed = seed, .S = S, .L = L, .M = M, .C = C, .dims = dims, .offs = offs,
               .out = out, .sigma = sigma, .next = 0};
  pthread_mutex_init(&J.mu, NULL);
  if (nthreads < 1) nthreads = 1;
  pthread_t *th = (pthread_t *)malloc(sizeof(pthread_t) * nthreads);
  for (int t = 1; t < nthreads; ++t) pthread_create(&th[t], NULL, lat_worker, &J);
  lat_worker(&J);
  for (int t = 1; t < nthreads; ++t) pthread_join(th[t], NULL);
  free(th);
  pthread_mutex_destroy(&J.mu);
}

/* Decoder weights, one decoder: W1[H][I], b1[H], {W[H][H], b[H]} x (layers-1),
 * Wout[C][H], bout[C].  Weights are Xavier-uniform U(-a, a) with
 * a = sqrt(6 / (fan_in + fan_out)); biases U(-1/sqrt(fan_in), 1/sqrt(fan_in)). */
void gen_decoder(uint64_t seed, uint32_t dec, uint32_t I, uint32_t H, uint32_t layers,
                 uint32_t C, float *dst) {
  uint64_t key = gen_key(seed, 2, dec, 0), i = 0;
  uint32_t fin = I, fout = H;
  for (uint32_t l = 0; l <= layers; ++l) {
    if (l == layers) fout = C;
    double a = sqrt(6.0 / (double)(fin + fout)), bb = 1.0 / sqrt((double)fin);
    for (uint64_t e = 0; e < (uint64_t)fin * fout; ++e) *dst++ = (float)(a * (2.0 * unif(key, i++) - 1.0));
    for (uint64_t e = 0; e < fout; ++e) *dst++ = (float)(bb * (2.0 * unif(key, i++) - 1.0));
    fin = H;
  }
}

/* A seeded Fisher-Yates permutation of 0..n-1. */
void gen_permutation(uint64_t seed, uint64_t tag, uint32_t n, uint32_t *out) {
  uint64_t key = gen_key(seed, 3, tag, 0);
  for (uint32_t i = 0; i < n; ++i) out[i] = i;
  for (uint32_t i = n; i > 1; --i) {
    uint32_t j = unif_int(key, n - i, i);
    uint32_t t = out[i - 1];
    out[i - 1] = out[j];
    out[j] = t;
  }
}

typedef struct {
  uint32_t set_id;
  float u, v, lod;
} gen_query;

/* n queries, set ~ U{0..S-1}, u, v ~ U[0,1) on the 2^-24 grid, lod = 0. */
void gen_queries_uniform(uint64_t seed, uint64_t n, uint32_t S, gen_query *out) {
  uint64_t key = gen_key(seed, 4, 0, 0);
  for (uint64_t i = 0; i < n; ++i) {
    out[i].set_id = unif_int(key, 3 * i, S);
    out[i].u = (float)(draw(key, 3 * i + 1) >> 40) * (1.0f / 16777216.0f);
    out[i].v = (float)(draw(key, 3 * i + 2) >> 40) * (1.0f / 16777216.0f);
    out[i].lod = 0.0f;
  }
}

/* Pixel (x, y) of a Ws x Hs screen in emission order: 8x4-pixel tiles in
 * row-major tile order, pixels row-major within a tile (one tile per warp). */
static uint64_t tile_order(uint32_t x, uint32_t y, uint32_t Ws) {
  uint32_t tiles_x = (Ws + 7) / 8;
  uint64_t tile = (uint64_t)(y / 4) * tiles_x + x / 8;
  return tile * 32 + (y % 4) * 8 + (x % 8);
}

/* Texel-centre raster of an N x N output for one set, emitted in 8x4 tiles.
 * N must be a multiple of 8 and of 4. */
void gen_queries_texel_centres(uint32_t N, uint32_t set_id, gen_query *out) {
  for (uint32_t y = 0; y < N; ++y)
    for (uint32_t x = 0; x < N; ++x) {
      gen_query *q = &out[tile_order(x, y, N)];
      q->set_id = set_id;
      q->u = ((float)x + 0.5f) / (float)N;
      q->v = ((float)y + 0.5f) / (float)N;
      q->lod = 0.0f;
    }
}

/* Controlled divergence: the raster above over S sets where every 32-query
 * warp holds exactly d distinct set ids (d <= 32, d <= S): d distinct sets are
 * drawn per warp, lanes take them round-robin, then the lanes are shuffled. */
void gen_queries_controlled(uint64_t seed, uint32_t N, uint32_t S, uint32_t d, gen_query *out) {
  gen_queries_texel_centres(N, 0, out);
  uint64_t nw = (uint64_t)N * N / 32;
  for (uint64_t w = 0; w < nw; ++w) {
    uint64_t key = gen_key(seed, 5, w, d), c = 0;
    uint32_t pool[1024], lanes[32];
    uint32_t S_ = S < 1024 ? S : 1024;
    for (uint32_t i = 0; i < S_; ++i) pool[i] = i;
    for (uint32_t i = 0; i < d; ++i) { /* partial Fisher-Yates: first d of pool */
      uint32_t j = i + unif_int(key, c++, S_ - i);
      uint32_t t = pool[i];
      pool[i] = pool[j];
      pool[j] = t;
    }
    for (uint32_t l = 0; l < 32; ++l) lanes[l] = pool[l % d];
    for (uint32_t i = 32; i > 1; --i) {
      uint32_t j = unif_int(key, c++, i);
      uint32_t t = lanes[i - 1];
      lanes[i - 1] = lanes[j];
      lanes[j] = t;
    }
    for (uint32_t l = 0; l < 32; ++l) out[w * 32 + l].set_id = lanes[l];
  }
}

/* ------------------------------------------------------------ G-buffer */

typedef struct {
  int64_t x, y;
  uint32_t set_id;
  double scale, c, s, ou, ov;
  float lod;
} region;

typedef struct {
  const region *R;
  uint32_t nR, Ws, Hs, cell, gw, gh;
  const uint32_t *cell_start, *cell_items;
  gen_query *out;
  uint32_t *labels;
  uint32_t next_row;
  pthread_mutex_t mu;
} vor_job;

/* Nearest site by squared integer distance; ties go to the lowest index. */
static uint32_t nearest(const vor_job *J, int64_t x, int64_t y) {
  int64_t cx = x / J->cell, cy = y / J->cell;
  int64_t best_d = INT64_MAX;
  uint32_t best = UINT32_MAX;
  for (int64_t r = 0;; ++r) {
    for (int64_t gy = cy - r; gy <= cy + r; ++gy) {
      if (gy < 0 || gy >= J->gh) continue;
      for (int64_t gx = cx - r; gx <= cx + r; ++gx) {
        if (gx < 0 || gx >= J->gw) continue;
        if (llabs(gx - cx) != r && llabs(gy - cy) != r) continue; /* ring only */
        uint32_t c = (uint32_t)(gy * J->gw + gx);
        for (uint32_t e = J->cell_start[c]; e < J->cell_start[c + 1]; ++e) {
          uint32_t k = J->cell_items[e];
          int64_t dx = x - J->R[k].x, dy = y - J->R[k].y, d2 = dx * dx + dy * dy;
          if (d2 < best_d || (d2 == best_d && k < best)) {
            best_d = d2;
            best = k;
          }
        }
      }
    }
    /* every site in ring r+1 or beyond is at least r*cell away */
    int64_t lim = r * (int64_t)J->cell;
    if (best != UINT32_MAX && best_d < lim * lim) return best;
    if (r > (int64_t)(J->gw + J->gh)) return best;
  }
}

static void *vor_worker(void *arg) {
  vor_job *J = (vor_job *)arg;
  for (;;) {
    pthread_mutex_lock(&J->mu);
    uint32_t y = J->next_row++;
    pthread_mutex_unlock(&J->mu);
    if (y >= J->Hs) break;
    for (uint32_t x = 0; x < J->Ws; ++x) {
      uint32_t k = nearest(J, x, y);
      const region *g = &J->R[k];
      double px = ((double)x + 0.5) / J->Ws, py = ((double)y + 0.5) / J->Ws;
      gen_query *q = &J->out[tile_order(x, y, J->Ws)];
      q->set_id = g->set_id;
      q->u = (float)(g->scale * (g->c * px - g->s * py) + g->ou);
      q->v = (float)(g->scale * (g->s * px + g->c * py) + g->ov);
      q->lod = g->lod;
      if (J->labels) J->labels[tile_order(x, y, J->Ws)] = k;
    }
  }
  return NULL;
}

/* One G-buffer frame: R Voronoi regions over a Ws x Hs screen, each with a set
 * id ~ U{0..S-1}, scale ~ U[1,8], rotation ~ U[0,2pi), offset ~ U[0,1)^2;
 * UV = scale * Rot * ((x+.5)/Ws, (y+.5)/Ws) + offset.  lod_mode 0: lod =
 * round(max(0, log2(scale * T / Ws))); lod_mode 1: lod ~ U[0, lod_max) per
 * region.  Queries are written in 8x4-tile order (Ws % 8 == 0, Hs % 4 == 0). */
void gen_gbuffer(uint64_t seed, uint32_t frame, uint32_t Ws, uint32_t Hs, uint32_t nR,
                 uint32_t S, uint32_t T, int lod_mode, float lod_max, gen_query *out,
                 uint32_t *labels, int nthreads) {
  region *R = (region *)malloc(sizeof(region) * nR);
  uint64_t key = gen_key(seed, 6, frame, 0);
  for (uint32_t k = 0; k < nR; ++k) {
    uint64_t b = 8ull * k;
    R[k].x = unif_int(key, b + 0, Ws);
    R[k].y = unif_int(key, b + 1, Hs);
    R[k].set_id = unif_int(key, b + 2, S);
    R[k].scale = 1.0 + 7.0 * unif(key, b + 3);
    double th = TWO_PI * unif(key, b + 4);
    R[k].c = cos(th);
    R[k].s = sin(th);
    R[k].ou = unif(key, b + 5);
    R[k].ov = unif(key, b + 6);
    if (lod_mode == 0) {
      double l = log2(R[k].scale * (double)T / (double)Ws);
      R[k].lod = (float)floor((l > 0.0 ? l : 0.0) + 0.5);
    } else {
      R[k].lod = (float)(lod_max * unif(key, b + 7));
    }
  }
  vor_job J;
  memset(&J, 0, sizeof J);
  J.R = R;
  J.nR = nR;
  J.Ws = Ws;
  J.Hs = Hs;
  double area = (double)Ws * Hs / (nR ? nR : 1);
  J.cell = (uint32_t)sqrt(area);
  if (J.cell < 4) J.cell = 4;
  J.gw = (Ws + J.cell - 1) / J.cell;
  J.gh = (Hs + J.cell - 1) / J.cell;
  uint32_t nc = J.gw * J.gh;
  uint32_t *start = (uint32_t *)calloc(nc + 1, sizeof(uint32_t));
  uint32_t *items = (uint32_t *)malloc(sizeof(uint32_t) * (nR ? nR : 1));
  uint32_t *fill = (uint32_t *)calloc(nc, sizeof(uint32_t));
  for (uint32_t k = 0; k < nR; ++k) start[(R[k].y / J.cell) * J.gw + R[k].x / J.cell + 1]++;
  for (uint32_t c = 0; c < nc; ++c) start[c + 1] += start[c];
  for (uint32_t k = 0; k < nR; ++k) { /* ascending k inside each cell */
    uint32_t c = (uint32_t)((R[k].y / J.cell) * J.gw + R[k].x / J.cell);
    items[start[c] + fill[c]++] = k;
  }
  J.cell_start = start;
  J.cell_items = items;
  J.out = out;
  J.labels = labels;
  pthread_mutex_init(&J.mu, NULL);
  if (nthreads < 1) nthreads = 1;
  pthread_t *th = (pthread_t *)malloc(sizeof(pthread_t) * nthreads);
  for (int t = 1; t < nthreads; ++t) pthread_create(&th[t], NULL, vor_worker, &J);
  vor_worker(&J);
  for (int t = 1; t < nthreads; ++t) pthread_join(th[t], NULL);
  pthread_mutex_destroy(&J.mu);
  free(th);
  free(start);
  free(items);
  free(fill);
  free(R);
}
