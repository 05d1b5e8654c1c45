// Internal declarations of libntc: the context, device helpers shared by the
// kernels (tap addressing, latent gather, mma.sync fragments) and launchers.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <climits>
#include <type_traits>

#include "../../include/ntc.h"

namespace ntc {

constexpr int kTile = NTC_TILE_ROWS;  // rows of one single-decoder tile
constexpr int kLevels = 2;            // latent grids per set
constexpr int kChannels = 8;          // fp16 channels per latent texel (16 B)
constexpr int kInDim = kLevels * kChannels;
constexpr int kMaxMips = 16;

// Base texel and dimensions of one (set, level, mip) grid.
struct alignas(16) GridDesc {
  unsigned long long base;
  uint32_t W, H;
};

// Device-side view of the assets, passed by value to kernels.
struct Assets {
  const uint4 *lat;         // latents, one uint4 (8 x fp16) per texel
  const GridDesc *grids;    // [num_sets][kLevels][num_mips]
  // Row-pair copy of the latents: texel (x, y) of a grid holds its own 8
  // channels and those of its right neighbour (x + 1 wrapped or clamped by the
  // address mode), 32 bytes, so one aligned load fetches both texels of a
  // bilinear row.  pgrids give each grid's base in `pair` (units of 32 bytes).
  const uint4 *pair;
  const GridDesc *pgrids;
  const uint32_t *map;      // [num_sets] set -> decoder
  uint32_t num_sets, num_decoders, num_mips, address_mode;
  // the decoder input (the general-shape kernels read these; the standard
  // kernels are compiled for 2 levels x 8 channels and no encoding)
  uint32_t num_levels = kLevels, channels = kChannels, pe_frequencies = 0;
};

// Per-decoder weight images.
//  mma image (fp16/bf16 bits, rows padded by 8 elements so ldmatrix is
//  conflict-free): W1[H][16+8], W2[H][H+8], W3[16][H+8] (rows >= C zero), then
//  fp32 biases b1[H], b2[H], b3[16].
//  fp32 image: W1[H][16], b1[H], W2[H][H], b2[H], W3[CP][H], b3[CP] (rows >= C
//  zero), CP = 8 or 16.
struct WeightImages {
  const uint8_t *mma;       // [D][mma_stride] bytes
  size_t mma_stride;
  const float *f32;         // [D][f32_stride] floats
  size_t f32_stride;
  const uint8_t *tc;        // [D][tc_stride] bytes, tcgen05 shared-memory image
  size_t tc_stride;
  const uint8_t *fma;       // [D][fma_stride] bytes, per-lane FMA image
  size_t fma_stride;
  uint32_t hidden, out_dim;
  uint32_t out_half;        // output rows in IEEE half (put_out) instead of fp32
};


inline __host__ __device__ size_t mma_image_bytes(uint32_t H) {
  return (size_t)H * (16 + 8) * 2 + (size_t)H * (H + 8) * 2 + (size_t)16 * (H + 8) * 2 +
         (size_t)(2 * H + 16) * 4;
}
inline __host__ __device__ uint32_t out_pad(uint32_t C) { return C <= 8 ? 8u : 16u; }
inline __host__ __device__ size_t f32_image_floats(uint32_t H, uint32_t C) {
  uint32_t CP = out_pad(C);
  return (size_t)H * 16 + H + (size_t)H * H + H + (size_t)CP * H + CP;
}
// Per-lane FMA image, element type T = the precision's operand type (fp32,
// fp16 or bf16): W1[H][16], W2[H][H], W3^T[H][CP] in T, then fp32 b1[H],
// b2[H], b3[CP] (rows of W3^T and entries of b3 at c >= C are zero).
inline __host__ __device__ size_t fma_image_bytes(uint32_t H, uint32_t C, uint32_t elem) {
  const size_t CP = out_pad(C);
  return ((size_t)H * 16 + (size_t)H * H + (size_t)H * CP) * elem + (2 * (size_t)H + CP) * 4;
}

// General decoder shapes (any shape ntc_create accepts besides the standard
// 2 x 8 latent channels -> 2 hidden layers of 64 or 128 with ReLU): inputs of
// num_levels x channels latents plus 4F positional-encoding values, 1..4
// hidden layers of 16..128, ReLU or LeakyReLU.
constexpr int kGenMaxIn = 64;      // in_dim limit
constexpr int kGenMaxHidden = 128;
constexpr int kGenMaxLayers = 4;   // hidden layers
constexpr int kGenMaxPe = 8;       // encoding frequencies

// Per-decoder images of a general shape.
//  tc image (fp16/bf16 tcgen05 B operands, no-swizzle K-major core matrices):
//    W1 [H][K1] (K1 = in_dim rounded up to 16, zero padded), W_l [H][H] for
//    each further hidden layer, Wout [16][H] (rows >= C zero), then fp32 b1[H],
//    b_l[H]..., bout[16], then the hidden biases again as fp16 (the fp16
//    epilogue adds them to the packed pair).
//  fma image (the precision's type T, row-major): W1 [H][in], W_l [H][H]...,
//    Wout^T [H][CP], then fp32 biases as above (bout padded to CP).
struct GenWeights {
  const uint8_t *tc;
  size_t tc_stride;
  const uint8_t *fma;
  size_t fma_stride;
  uint32_t in_dim, k1, hidden, layers, out_dim, activation;
  float slope;
  uint32_t out_half;  // output rows in IEEE half (put_out) instead of fp32
};

inline __host__ __device__ uint32_t gen_k1(uint32_t in_dim) { return (in_dim + 15) / 16 * 16; }
inline __host__ __device__ size_t gen_tc_weight_bytes(uint32_t in_dim, uint32_t H, uint32_t layers) {
  return ((size_t)H * gen_k1(in_dim) + (size_t)(layers - 1) * H * H + (size_t)16 * H) * 2;
}
inline __host__ __device__ size_t gen_bias_floats(uint32_t H, uint32_t layers) {
  return (size_t)layers * H + 16;
}
inline __host__ __device__ size_t gen_tc_image_bytes(uint32_t in_dim, uint32_t H, uint32_t layers) {
  return gen_tc_weight_bytes(in_dim, H, layers) + gen_bias_floats(H, layers) * 4 + (size_t)layers * H * 2;
}
inline __host__ __device__ size_t gen_fma_image_bytes(uint32_t in_dim, uint32_t H, uint32_t layers, uint32_t C,
                                                      uint32_t elem) {
  const size_t CP = out_pad(C);
  const size_t w = ((size_t)H * in_dim + (size_t)(layers - 1) * H * H + (size_t)H * CP) * elem;
  return (w + 15) / 16 * 16 + ((size_t)layers * H + CP) * 4;
}

// Bucketing results on the device: row i of the bucketed order is query
// perm[i] of the caller's array; when the bucketing copied the records
// (meta[meta_copied(D)] != 0) that record is also sorted[i].  identity_n != 0:
// one decoder and no sorting, row i is query i of `queries` (identity_n
// queries); sorted, perm and meta are unused.
struct Buckets {
  const ntc_query *queries;  // the caller's queries, in their own order
  const ntc_query *sorted;   // the query records in (decoder, index) order, if copied
  const uint32_t *perm;      // original index of each row
  const uint32_t *meta;      // [0] num_tiles, seg_start[D+2], tile_start[D+2], copied, divergence
  uint32_t identity_n = 0;
};
inline __host__ __device__ uint32_t meta_words(uint32_t D) { return 1 + 2 * (D + 2) + 2; }
// meta[meta_copied(D)]: 1 when the bucketing wrote the query records in bucket
// order (Buckets::sorted); 0 when the decode reads query perm[i] of the
// caller's array
inline __host__ __device__ uint32_t meta_copied(uint32_t D) { return 1 + 2 * (D + 2); }
// meta[meta_divergence(D)]: the call's sum over groups of 32 consecutive
// queries of (distinct decoders in the group - 1), Eq. 1's numerator
inline __host__ __device__ uint32_t meta_divergence(uint32_t D) { return 2 + 2 * (D + 2); }
// The bucketing copies the records when Eq. 1's score (the mean over 32-query
// groups of distinct decoders - 1) exceeds this: the queries of one decoder
// are then scattered over the array, and reading them through perm would
// touch each sector once per decoder
constexpr uint32_t kCopyAboveScore = 4;

// ------------------------------------------------------------- device helpers

// Programmatic dependent launch: a kernel launched with launch_pdl may start
// while its predecessor on the stream is still running; pdl_wait() blocks
// until that predecessor has completed and its writes are visible (a no-op for
// an ordinary launch).  pdl_trigger() lets the successor start launching.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }


// One axis of the tap addressing, fp32 round-to-nearest with no contraction.
__device__ __forceinline__ void axis_taps(float c, uint32_t n, uint32_t mode, uint32_t &i0,
                                          uint32_t &i1, float &frac) {
  float x;
  if (mode == 0) {
    float cw = __fsub_rn(c, floorf(c));
    x = __fsub_rn(__fmul_rn(cw, (float)n), 0.5f);
  } else {
    x = __fsub_rn(__fmul_rn(c, (float)n), 0.5f);
  }
  float x0f = floorf(x);
  frac = __fsub_rn(x, x0f);
  if (mode == 0) {
    int x0 = (int)x0f;  // in [-1, n-1]
    i0 = x0 < 0 ? n - 1 : (uint32_t)x0;
    uint32_t a1 = (uint32_t)(x0 + 1);
    i1 = a1 >= n ? a1 - n : a1;
  } else {
    int x0 = (int)fminf(fmaxf(x0f, -1.0f), (float)n);
    int hi = (int)n - 1;
    i0 = (uint32_t)min(max(x0, 0), hi);
    i1 = (uint32_t)min(max(x0 + 1, 0), hi);
  }
}

// Texel indices and bilinear weights of one grid (tap order 00, 10, 01, 11).
__device__ __forceinline__ void grid_taps(const GridDesc &g, float u, float v, uint32_t mode,
                                          unsigned long long idx[4], float w[4]) {
  uint32_t i0, i1, j0, j1;
  float wx, wy;
  axis_taps(u, g.W, mode, i0, i1, wx);
  axis_taps(v, g.H, mode, j0, j1, wy);
  unsigned long long r0 = g.base + (unsigned long long)j0 * g.W;
  unsigned long long r1 = g.base + (unsigned long long)j1 * g.W;
  idx[0] = r0 + i0;
  idx[1] = r0 + i1;
  idx[2] = r1 + i0;
  idx[3] = r1 + i1;
  float ax = __fsub_rn(1.0f, wx), ay = __fsub_rn(1.0f, wy);
  w[0] = __fmul_rn(ax, ay);
  w[1] = __fmul_rn(wx, ay);
  w[2] = __fmul_rn(ax, wy);
  w[3] = __fmul_rn(wx, wy);
}

__device__ __forceinline__ bool query_bad(const Assets &A, const ntc_query &q) {
  return q.set_id >= A.num_sets || !isfinite(q.u) || !isfinite(q.v);
}

// Mip selection: lo and blend t (t > 0 only when mip lo+1 exists).
__device__ __forceinline__ int select_mip(float lod, uint32_t num_mips, float &t) {
  float lam = fmaxf(lod, 0.0f);
  float lof = fminf(floorf(lam), (float)(num_mips - 1));
  int lo = (int)lof;
  t = (lo == (int)num_mips - 1) ? 0.0f : __fsub_rn(lam, lof);
  return lo;
}

__device__ __forceinline__ void accum_tap(float f[kChannels], uint4 raw, float w) {
  const __half2 *h = reinterpret_cast<const __half2 *>(&raw);
#pragma unroll
  for (int p = 0; p < 4; ++p) {
    float2 x = __half22float2(h[p]);
    f[2 * p] = fmaf(w, x.x, f[2 * p]);
    f[2 * p + 1] = fmaf(w, x.y, f[2 * p + 1]);
  }
}

// The fp32 MLP input of a (good) query: f[0..7] level 0, f[8..15] level 1.
// All tap loads of a query are issued before any is consumed.
__device__ __forceinline__ void query_features(const Assets &A, const ntc_query &q,
                                               float f[kInDim]) {
  float t;
  int lo = select_mip(q.lod, A.num_mips, t);
  const GridDesc *g = A.grids + (size_t)q.set_id * kLevels * A.num_mips;
#pragma unroll
  for (int c = 0; c < kInDim; ++c) f[c] = 0.0f;
  if (t == 0.0f) {
    unsigned long long idx[kLevels][4];
    float w[kLevels][4];
    uint4 raw[kLevels][4];
#pragma unroll
    for (int k = 0; k < kLevels; ++k) grid_taps(g[k * A.num_mips + lo], q.u, q.v, A.address_mode, idx[k], w[k]);
#pragma unroll
    for (int k = 0; k < kLevels; ++k)
#pragma unroll
      for (int p = 0; p < 4; ++p) raw[k][p] = __ldg(A.lat + idx[k][p]);
#pragma unroll
    for (int k = 0; k < kLevels; ++k)
#pragma unroll
      for (int p = 0; p < 4; ++p) accum_tap(f + k * kChannels, raw[k][p], w[k][p]);
  } else {
    float s = __fsub_rn(1.0f, t);
#pragma unroll
    for (int k = 0; k < kLevels; ++k) {
      unsigned long long idx[2][4];
      float w[2][4];
      uint4 raw[2][4];
      grid_taps(g[k * A.num_mips + lo], q.u, q.v, A.address_mode, idx[0], w[0]);
      grid_taps(g[k * A.num_mips + lo + 1], q.u, q.v, A.address_mode, idx[1], w[1]);
#pragma unroll
      for (int m = 0; m < 2; ++m)
#pragma unroll
        for (int p = 0; p < 4; ++p) raw[m][p] = __ldg(A.lat + idx[m][p]);
#pragma unroll
      for (int p = 0; p < 4; ++p) accum_tap(f + k * kChannels, raw[0][p], w[0][p] * s);
#pragma unroll
      for (int p = 0; p < 4; ++p) accum_tap(f + k * kChannels, raw[1][p], w[1][p] * t);
    }
  }
}

// Positional encoding of one coordinate pair at input offset BASE: for k < F,
// sin / cos of 2 pi 2^k u and of 2 pi 2^k v (u, v as the taps see them).  One
// sincospif per coordinate gives k = 0; every further frequency doubles the
// angle (sin 2a = 2 sin a cos a, cos 2a = cos^2 a - sin^2 a), which keeps the
// error within a few ulp for the at most 8 frequencies.
template <int BASE, int N>
__device__ __forceinline__ void pe_features(float u, float v, uint32_t F, float (&f)[N]) {
  if (F == 0) return;
  float su, cu, sv, cv;
  sincospif(2.0f * u, &su, &cu);
  sincospif(2.0f * v, &sv, &cv);
#pragma unroll
  for (int k = 0; k < kGenMaxPe; ++k) {
    if (BASE + 4 * k + 3 >= N) break;
    if (k < (int)F) {
      f[BASE + 4 * k + 0] = su;
      f[BASE + 4 * k + 1] = cu;
      f[BASE + 4 * k + 2] = sv;
      f[BASE + 4 * k + 3] = cv;
      const float su2 = 2.0f * su * cu, cu2 = cu * cu - su * su;
      const float sv2 = 2.0f * sv * cv, cv2 = cv * cv - sv * sv;
      su = su2, cu = cu2, sv = sv2, cv = cv2;
    }
  }
}

// The latent features of level K of a good query, C channels per texel, at
// input offset K * C; with t > 0 the two mips are blended (weights scaled by
// 1 - t and t, as in query_features).  Every tap load of the level (both mips)
// is issued before any is consumed.
template <int K, int C, int N>
__device__ __forceinline__ void gen_level(const Assets &A, const GridDesc *g, int lo, float t, const ntc_query &q,
                                          float (&f)[N]) {
  using Raw = typename std::conditional<C == 8, uint4, uint2>::type;
  const bool two = t > 0.0f;
  unsigned long long idx[2][4];
  float w[2][4];
  grid_taps(g[K * A.num_mips + lo], q.u, q.v, A.address_mode, idx[0], w[0]);
  if (two) grid_taps(g[K * A.num_mips + lo + 1], q.u, q.v, A.address_mode, idx[1], w[1]);
  Raw raw[2][4];
#pragma unroll
  for (int m = 0; m < 2; ++m)
#pragma unroll
    for (int p = 0; p < 4; ++p)
      if (m == 0 || two) raw[m][p] = __ldg(reinterpret_cast<const Raw *>(A.lat) + idx[m][p]);
#pragma unroll
  for (int m = 0; m < 2; ++m) {
    if (m == 1 && !two) break;
    const float s = !two ? 1.0f : (m == 0 ? __fsub_rn(1.0f, t) : t);
#pragma unroll
    for (int p = 0; p < 4; ++p) {
      const float wp = !two ? w[m][p] : w[m][p] * s;
      const __half2 *h = reinterpret_cast<const __half2 *>(&raw[m][p]);
#pragma unroll
      for (int c = 0; c < C / 2; ++c) {
        const float2 x = __half22float2(h[c]);
        f[K * C + 2 * c] = fmaf(wp, x.x, f[K * C + 2 * c]);
        f[K * C + 2 * c + 1] = fmaf(wp, x.y, f[K * C + 2 * c + 1]);
      }
    }
  }
}

// The MLP input of a good query for a general shape with L levels of C
// channels: the latent features, then the positional encoding; zero up to N.
// grids: A.grids, or a copy of it (in shared memory).
template <int L, int C, int N>
__device__ __forceinline__ void gen_features_t(const Assets &A, const GridDesc *grids, const ntc_query &q,
                                               float (&f)[N]) {
  static_assert(N >= L * C + 4 * kGenMaxPe && N <= kGenMaxIn, "feature array too small");
#pragma unroll
  for (int i = 0; i < N; ++i) f[i] = 0.0f;
  float t;
  const int lo = select_mip(q.lod, A.num_mips, t);
  const GridDesc *g = grids + (size_t)q.set_id * L * A.num_mips;
  const float u = A.address_mode == 0 ? __fsub_rn(q.u, floorf(q.u)) : q.u;
  const float v = A.address_mode == 0 ? __fsub_rn(q.v, floorf(q.v)) : q.v;
  gen_level<0, C, N>(A, g, lo, t, q, f);
  if (L == 2) gen_level<1, C, N>(A, g, lo, t, q, f);
  pe_features<L * C, N>(u, v, A.pe_frequencies, f);
}

// Only the latent features of a good query: L levels of C channels.
template <int L, int C>
__device__ __forceinline__ void gen_latents_t(const Assets &A, const GridDesc *grids, const ntc_query &q,
                                              float (&f)[L * C]) {
#pragma unroll
  for (int i = 0; i < L * C; ++i) f[i] = 0.0f;
  float t;
  const int lo = select_mip(q.lod, A.num_mips, t);
  const GridDesc *g = grids + (size_t)q.set_id * L * A.num_mips;
  gen_level<0, C, L * C>(A, g, lo, t, q, f);
  if (L == 2) gen_level<1, C, L * C>(A, g, lo, t, q, f);
}

// The latent features of a good query in packed fp16 pairs, h[i] = channels
// (2i, 2i+1) of the L x C inputs: the tensor-core path's blend (hfma2 on the
// fp16 latents; every tap load of a level is issued before any is consumed).
template <int L, int C>
__device__ __forceinline__ void gen_latents_h2(const Assets &A, const GridDesc *grids, const ntc_query &q,
                                               __half2 (&h)[L * C / 2]) {
  using Raw = typename std::conditional<C == 8, uint4, uint2>::type;
#pragma unroll
  for (int i = 0; i < L * C / 2; ++i) h[i] = __float2half2_rn(0.0f);
  float t;
  const int lo = select_mip(q.lod, A.num_mips, t);
  const GridDesc *g = grids + (size_t)q.set_id * L * A.num_mips;
  const bool two = t > 0.0f;
#pragma unroll
  for (int k = 0; k < L; ++k) {
    unsigned long long idx[2][4];
    float w[2][4];
    grid_taps(g[k * A.num_mips + lo], q.u, q.v, A.address_mode, idx[0], w[0]);
    if (two) grid_taps(g[k * A.num_mips + lo + 1], q.u, q.v, A.address_mode, idx[1], w[1]);
    Raw raw[2][4];
#pragma unroll
    for (int m = 0; m < 2; ++m)
#pragma unroll
      for (int p = 0; p < 4; ++p)
        if (m == 0 || two) raw[m][p] = __ldg(reinterpret_cast<const Raw *>(A.lat) + idx[m][p]);
#pragma unroll
    for (int m = 0; m < 2; ++m) {
      if (m == 1 && !two) break;
      const float s = !two ? 1.0f : (m == 0 ? __fsub_rn(1.0f, t) : t);
#pragma unroll
      for (int p = 0; p < 4; ++p) {
        const __half2 ww = __float2half2_rn(!two ? w[m][p] : w[m][p] * s);
        const __half2 *x = reinterpret_cast<const __half2 *>(&raw[m][p]);
#pragma unroll
        for (int c = 0; c < C / 2; ++c) h[k * C / 2 + c] = __hfma2(ww, x[c], h[k * C / 2 + c]);
      }
    }
  }
}

// The coordinates the taps see (the positional encoding's input).
__device__ __forceinline__ void pe_coords(const Assets &A, const ntc_query &q, float &u, float &v) {
  u = A.address_mode == 0 ? __fsub_rn(q.u, floorf(q.u)) : q.u;
  v = A.address_mode == 0 ? __fsub_rn(q.v, floorf(q.v)) : q.v;
}

// Any general shape, dispatched at run time (kGenMaxIn values).
__device__ __forceinline__ void gen_features(const Assets &A, const GridDesc *grids, const ntc_query &q,
                                             float (&f)[kGenMaxIn]) {
  if (A.channels == 8) {
    if (A.num_levels == 2) gen_features_t<2, 8, kGenMaxIn>(A, grids, q, f);
    else gen_features_t<1, 8, kGenMaxIn>(A, grids, q, f);
  } else {
    if (A.num_levels == 2) gen_features_t<2, 4, kGenMaxIn>(A, grids, q, f);
    else gen_features_t<1, 4, kGenMaxIn>(A, grids, q, f);
  }
}

__device__ __forceinline__ ntc_query load_query(const ntc_query *q) {
  uint4 r = __ldg(reinterpret_cast<const uint4 *>(q));
  ntc_query out;
  out.set_id = r.x;
  out.u = __uint_as_float(r.y);
  out.v = __uint_as_float(r.z);
  out.lod = __uint_as_float(r.w);
  return out;
}

// Whether the query records of this launch's bucketing were copied (read
// once the bucketing has finished; false without bucketing).
__device__ __forceinline__ bool rows_copied(const Buckets &B, uint32_t D) {
  return !B.identity_n && __ldg(B.meta + meta_copied(D)) != 0u;
}

// Row `pos` of the bucketed order: its output row (original index) and query.
__device__ __forceinline__ void bucket_row(const Buckets &B, bool copied, uint32_t pos, uint32_t &oi, ntc_query &q) {
  oi = B.identity_n ? pos : __ldg(B.perm + pos);
  q = load_query(copied ? B.sorted + pos : B.queries + oi);
}

// Tile t of the bucketed order: decoder, first sorted position and length.
__device__ __forceinline__ void tile_info(const uint32_t *meta, uint32_t D, uint32_t t,
                                          uint32_t &dec, uint32_t &start, uint32_t &len) {
  const uint32_t *seg = meta + 1;           // seg_start[D+2]
  const uint32_t *tst = meta + 1 + (D + 2); // tile_start[D+2]
  // largest d in [0, D] with tile_start[d] <= t
  uint32_t lo = 0, hi = D + 1;
  while (hi - lo > 1) {
    uint32_t mid = (lo + hi) >> 1;
    if (__ldg(tst + mid) <= t) lo = mid; else hi = mid;
  }
  dec = lo;
  start = __ldg(seg + lo) + (t - __ldg(tst + lo)) * kTile;
  uint32_t end = __ldg(seg + lo + 1);
  len = min((uint32_t)kTile, end - start);
}

// The tiles of one role in increasing order: the decoder index only moves
// forward, so a lookup is a few compares instead of a binary search.  With
// ident_n != 0 (one decoder, nothing sorted) tile t is queries 128t .. of the
// caller's array.
// One output value in the context's output format: fp32, or IEEE half rounded
// to nearest even (the fp16 output of Sec. 4.4's fp16 kernels); a bad query's
// row is NaN in every channel.
__device__ __forceinline__ void put_out(void *out, size_t i, float y, bool half) {
  if (half)
    reinterpret_cast<__half *>(out)[i] = __float2half_rn(y);
  else
    reinterpret_cast<float *>(out)[i] = y;
}
__device__ __forceinline__ void put_nan_row(void *out, size_t row, uint32_t C, bool half) {
  for (uint32_t c = 0; c < C; ++c) {
    if (half)
      reinterpret_cast<unsigned short *>(out)[row * C + c] = 0x7E00u;
    else
      reinterpret_cast<float *>(out)[row * C + c] = __int_as_float(0x7fc00000);
  }
}

struct TileWalk {
  uint32_t d = 0;
  uint32_t ident_n = 0;
  __device__ __forceinline__ void at(const uint32_t *seg, const uint32_t *tst, uint32_t D, uint32_t t,
                                     uint32_t &dec, uint32_t &start, uint32_t &len) {
    if (ident_n) {
      dec = 0;
      start = t * kTile;
      len = min((uint32_t)kTile, ident_n - start);
      return;
    }
    while (d < D && tst[d + 1] <= t) ++d;
    dec = d;
    start = seg[d] + (t - tst[d]) * kTile;
    len = min((uint32_t)kTile, seg[d + 1] - start);
  }
};

// ---------------------------------------------------------------- launchers

// Device scratch of one bucketing call.
struct Scratch {
  uint32_t *perm;     // [n]
  ntc_query *sorted;  // [n] the query records in bucket order
  uint32_t *meta;     // bucket_meta_words(D): the tile table, then the totals
                      // [D+1], a ticket and the divergence sum (zero between
                      // calls)
  uint32_t *counts;   // [bucket_count_words(D, n)] per-chunk counts (k_count)
  uint32_t *offs;     // [bucket_count_words(D, n)] per-chunk offsets (k_scan);
                      // a separate array, so that running k_scan again (a
                      // profiler's replay) reads the same counts
  void *dec;          // [n] decoder per query, bucket_dec_bytes(D) bytes each;
                      // null: k_place reads the decoders from the records, which
                      // it then always stages and copies (copy must be 1)
};

constexpr int kBucketThreads = 256;
constexpr int kBucketItems = 8;  // queries per thread
constexpr int kBucketChunk = kBucketThreads * kBucketItems;
size_t bucket_chunks(size_t n);
size_t bucket_count_words(uint32_t D, size_t n);
size_t bucket_meta_words(uint32_t D);
size_t bucket_dec_bytes(uint32_t D);

// copy: 0 = copy the records when Eq. 1's score exceeds kCopyAboveScore, 1 =
// always copy them
cudaError_t launch_bucket(const Assets &A, const ntc_query *q, size_t n, const Scratch &s, cudaStream_t st,
                          int *launches, int copy = 0);
cudaError_t launch_tiles_export(const uint32_t *meta, uint32_t D, uint32_t *tiles, uint32_t *num_tiles,
                                uint32_t *counts, size_t max_tiles, cudaStream_t st, int *launches);
cudaError_t launch_decode_fp32(const Assets &A, const WeightImages &W, const Buckets &B, size_t n,
                               float *out, unsigned long long *err, int num_sms, cudaStream_t st,
                               int *launches);
cudaError_t launch_decode_mma(const Assets &A, const WeightImages &W, const Buckets &B, size_t n,
                              float *out, unsigned long long *err, bool bf16, int num_sms,
                              cudaStream_t st, int *launches);
cudaError_t launch_decode_divergent(const Assets &A, const WeightImages &W, const ntc_query *q,
                                    size_t n, float *out, unsigned long long *err, bool bf16,
                                    int num_sms, cudaStream_t st, int *launches);
cudaError_t launch_decode_divergent_fma(const Assets &A, const WeightImages &W, const ntc_query *q,
                                        size_t n, float *out, unsigned long long *err, ntc_precision prec,
                                        int num_sms, cudaStream_t st, int *launches);
cudaError_t launch_pack_fma(const float *w32, uint32_t D, uint32_t H, uint32_t C, ntc_precision prec,
                            uint8_t *fma, size_t fma_stride, cudaStream_t st);
// General shapes: the tcgen05 decode over bucketed tiles, and the per-lane
// FMA decode over the queries in bucket order (B non-null) or in their own
// order (B null).
cudaError_t launch_decode_gen_tc(const Assets &A, const GenWeights &G, const Buckets &B, size_t n, void *out,
                                 unsigned long long *err, unsigned int *status, bool bf16, int num_sms,
                                 cudaStream_t st, int *launches);
cudaError_t launch_decode_gen_fma(const Assets &A, const GenWeights &G, const Buckets *B, const ntc_query *q,
                                  size_t n, float *out, unsigned long long *err, ntc_precision prec, int num_sms,
                                  cudaStream_t st, int *launches);
cudaError_t launch_pack_gen(const float *w32, uint32_t D, const GenWeights &G, ntc_precision prec, uint8_t *tc,
                            uint8_t *fma, cudaStream_t st);
cudaError_t launch_decode_tc(const Assets &A, const WeightImages &W, const Buckets &B, size_t n,
                             void *out, unsigned long long *err, unsigned int *status, bool bf16,
                             int num_sms, cudaStream_t st, int *launches);
cudaError_t launch_decode_tc_debug(const Assets &A, const WeightImages &W, const Buckets &B, size_t n,
                                   void *out, unsigned long long *err, unsigned int *status, bool bf16,
                                   int num_sms, cudaStream_t st, int *launches, ntc_debug_row *rows);
cudaError_t launch_pack_tc(const float *w32, uint32_t D, uint32_t H, uint32_t C, bool bf16,
                           uint8_t *tc, size_t tc_stride, cudaStream_t st);
cudaError_t launch_debug_taps(const Assets &A, const ntc_query *q, size_t n, unsigned long long *idx,
                              float *w, float *t, cudaStream_t st, int *launches);
cudaError_t launch_debug_features(const Assets &A, const ntc_query *q, size_t n, float *f,
                                  cudaStream_t st, int *launches);
// CTAs of `kernel` that fit on one SM at once (threads, registers, shared
// memory), computed from the kernel's own attributes and the device's limits.
template <typename Kernel>
inline int resident_ctas(Kernel kernel, int threads, size_t dyn_smem) {
  cudaFuncAttributes fa;
  if (cudaFuncGetAttributes(&fa, kernel) != cudaSuccess) return 1;
  int dev = 0, regs_sm = 65536, smem_sm = 233472, thr_sm = 2048, cta_sm = 32;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&regs_sm, cudaDevAttrMaxRegistersPerMultiprocessor, dev);
  cudaDeviceGetAttribute(&smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev);
  cudaDeviceGetAttribute(&thr_sm, cudaDevAttrMaxThreadsPerMultiProcessor, dev);
  cudaDeviceGetAttribute(&cta_sm, cudaDevAttrMaxBlocksPerMultiprocessor, dev);
  const int warps = (threads + 31) / 32;
  const int regs_cta = warps * ((fa.numRegs + 7) / 8 * 8) * 32;  // 256-register allocation units per warp
  int occ = regs_cta > 0 ? regs_sm / regs_cta : cta_sm;
  occ = occ < thr_sm / (warps * 32) ? occ : thr_sm / (warps * 32);
  const size_t smem_cta = dyn_smem + fa.sharedSizeBytes + 1024;  // 1 KB per CTA reserved by the system
  const int by_smem = (int)((size_t)smem_sm / smem_cta);
  occ = occ < by_smem ? occ : by_smem;
  occ = occ < cta_sm ? occ : cta_sm;
  return occ < 1 ? 1 : occ;
}

// Per-device one-time set-up.  Kernel attributes (the dynamic shared-memory
// limit, the carveout) belong to a device, so every device a process uses
// needs its own; once() runs f on the current device the first time that
// device asks and remembers success, value() caches an int result (an
// occupancy) per device.  Threads racing on a first use may both run f, which
// must therefore be idempotent.
class PerDevice {
 public:
  PerDevice() {
    for (auto &v : val_) v.store(INT_MIN, std::memory_order_relaxed);
  }
  template <typename F>
  cudaError_t once(F f) {
    std::atomic<int> *slot = slot_of();
    if (slot && slot->load(std::memory_order_acquire) == 0) return cudaSuccess;
    const cudaError_t e = f();
    if (e == cudaSuccess && slot) slot->store(0, std::memory_order_release);
    return e;
  }
  template <typename F>
  int value(F f) {
    std::atomic<int> *slot = slot_of();
    if (slot) {
      const int v = slot->load(std::memory_order_acquire);
      if (v != INT_MIN) return v;
    }
    const int v = f();
    if (slot) slot->store(v, std::memory_order_release);
    return v;
  }

 private:
  static constexpr int kMaxDevices = 64;
  std::atomic<int> val_[kMaxDevices];
  std::atomic<int> *slot_of() {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
    return &val_[dev];
  }
};

// False when the environment variable NTC_NO_PDL is set (read once per
// process): launch_pdl then makes ordinary launches, which start only after
// their predecessor has ended.  The results are the same; a profiler that
// replays one kernel of the chain needs it.
bool pdl_enabled();

// Launch with programmatic stream serialisation (see pdl_wait).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                       Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = pdl_enabled() ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

cudaError_t launch_build_pairs(const Assets &A, const uint32_t *chunk_grid, const uint32_t *chunk_start,
                               uint32_t num_chunks, uint4 *pair, cudaStream_t st);
constexpr uint32_t kPairChunk = 65536;  // texels per work item of launch_build_pairs
cudaError_t launch_pack_weights(const float *w32, uint32_t D, uint32_t H, uint32_t C, bool bf16,
                                uint8_t *mma, size_t mma_stride, float *f32, size_t f32_stride,
                                uint8_t *tc, size_t tc_stride, cudaStream_t st);
size_t tc_image_bytes(uint32_t H);

}  // namespace ntc
