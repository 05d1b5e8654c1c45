// Clustered map source: k-means over per-texture embeddings (Alg. 2, Stage 2).
//
// The paper clusters the textures' CLIP embeddings F [n][512] into m groups with
// k-means and gives every group one shared decoder; at run time only the
// resulting set -> decoder map c(i) matters.  ntc_kmeans_map computes that map
// on the GPU with Lloyd's iteration, deterministically:
//   start       mu_g = F[init[g]]
//   assignment  c(i) = argmin_g sum_j (F[i][j] - mu_g[j])^2, fp64, j increasing,
//               ties to the smallest g (one warp per embedding, lanes over g)
//   update      mu_g[j] = (sum over i increasing with c(i) = g of F[i][j]) / |g|
//               (one thread per (g, j)); an empty group keeps its centroid
//   stop        when no assignment changes, or after max_iters assignments.
// Every fp64 operation is an explicit round-to-nearest add, subtract, multiply
// or divide with no contraction, in a fixed order, so the map and the
// centroids do not depend on the launch shape.
#include <algorithm>
#include <vector>

#include "ntc_internal.cuh"

namespace ntc {
void set_last_error(const char *msg);
}

using namespace ntc;

namespace {

__global__ void k_km_assign(const double *F, const double *mu, uint32_t n, uint32_t dim, uint32_t m,
                            uint32_t *map, unsigned int *changed) {
  const uint32_t lane = threadIdx.x & 31;
  const size_t warps = (size_t)gridDim.x * (blockDim.x / 32);
  for (size_t i = (size_t)blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5); i < n; i += warps) {
    const double *x = F + i * dim;
    double best_d = 0.0;
    uint32_t best = 0xFFFFFFFFu;
    for (uint32_t g = lane; g < m; g += 32) {
      const double *c = mu + (size_t)g * dim;
      double dist = 0.0;
      for (uint32_t j = 0; j < dim; ++j) {
        const double d = __dsub_rn(x[j], c[j]);
        dist = __dadd_rn(dist, __dmul_rn(d, d));
      }
      if (best == 0xFFFFFFFFu || dist < best_d) {  // g increases: ties keep the smaller g
        best_d = dist;
        best = g;
      }
    }
    // warp argmin: smaller distance, then smaller group index
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const double od = __shfl_down_sync(0xFFFFFFFFu, best_d, o);
      const uint32_t og = __shfl_down_sync(0xFFFFFFFFu, best, o);
      if (og != 0xFFFFFFFFu && (best == 0xFFFFFFFFu || od < best_d || (od == best_d && og < best))) {
        best_d = od;
        best = og;
      }
    }
    if (lane == 0) {
      if (map[i] != best) atomicAdd(changed, 1u);
      map[i] = best;
    }
  }
}

__global__ void k_km_update(const double *F, const uint32_t *map, uint32_t n, uint32_t dim, uint32_t m,
                            double *mu) {
  const size_t total = (size_t)m * dim;
  for (size_t e = (size_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (size_t)gridDim.x * blockDim.x) {
    const uint32_t g = (uint32_t)(e / dim), j = (uint32_t)(e % dim);
    double s = 0.0;
    uint32_t count = 0;
    for (uint32_t i = 0; i < n; ++i)
      if (map[i] == g) {
        s = __dadd_rn(s, F[(size_t)i * dim + j]);
        ++count;
      }
    if (count) mu[e] = __ddiv_rn(s, (double)count);
  }
}

ntc_status km_fail(ntc_status s, const char *m) {
  set_last_error(m);
  return s;
}

struct DevBuf {
  void *p = nullptr;
  ~DevBuf() {
    if (p) cudaFree(p);
  }
};

}  // namespace

extern "C" NTC_API ntc_status ntc_kmeans_map(const float *h_features, uint32_t n, uint32_t dim, uint32_t m,
                                             const uint32_t *h_init, uint32_t max_iters, uint32_t *h_map,
                                             double *h_centroids, uint32_t *iters_run) {
  if (!h_features || !h_init || !h_map) return km_fail(NTC_ERR_INVALID_ARG, "null host pointer");
  if (n < 1 || n > (1u << 24)) return km_fail(NTC_ERR_INVALID_ARG, "n must be in 1..2^24");
  if (dim < 1 || dim > 4096) return km_fail(NTC_ERR_INVALID_ARG, "dim must be in 1..4096");
  if (m < 1 || m > n || m > NTC_MAX_DECODERS)
    return km_fail(NTC_ERR_INVALID_ARG, "m must be in 1..min(n, 4095)");
  if (max_iters < 1) return km_fail(NTC_ERR_INVALID_ARG, "max_iters must be >= 1");
  std::vector<uint8_t> seen(n, 0);
  for (uint32_t g = 0; g < m; ++g) {
    if (h_init[g] >= n || seen[h_init[g]]) return km_fail(NTC_ERR_INVALID_ARG, "init must hold m distinct rows < n");
    seen[h_init[g]] = 1;
  }
  const size_t nf = (size_t)n * dim;
  std::vector<double> F(nf), mu((size_t)m * dim);
  for (size_t e = 0; e < nf; ++e) {
    const float v = h_features[e];
    if (!(v == v) || v - v != 0.0f) return km_fail(NTC_ERR_INVALID_ARG, "features must be finite");
    F[e] = (double)v;
  }
  for (uint32_t g = 0; g < m; ++g)
    for (uint32_t j = 0; j < dim; ++j) mu[(size_t)g * dim + j] = F[(size_t)h_init[g] * dim + j];
  DevBuf dF, dmu, dmap, dchg;
  cudaError_t e = cudaMalloc(&dF.p, nf * 8);
  if (e == cudaSuccess) e = cudaMalloc(&dmu.p, mu.size() * 8);
  if (e == cudaSuccess) e = cudaMalloc(&dmap.p, (size_t)n * 4);
  if (e == cudaSuccess) e = cudaMalloc(&dchg.p, 4);
  if (e == cudaSuccess) e = cudaMemcpy(dF.p, F.data(), nf * 8, cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemcpy(dmu.p, mu.data(), mu.size() * 8, cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemset(dmap.p, 0xFF, (size_t)n * 4);
  if (e != cudaSuccess)
    return km_fail(e == cudaErrorMemoryAllocation ? NTC_ERR_OUT_OF_MEMORY : NTC_ERR_CUDA, cudaGetErrorString(e));
  int sms = 1;
  int dev = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const unsigned ablocks = (unsigned)std::min<size_t>(((size_t)n + 7) / 8, (size_t)sms * 8);
  const unsigned ublocks = (unsigned)std::min<size_t>(((size_t)m * dim + 255) / 256, (size_t)sms * 8);
  uint32_t t = 0;
  while (t < max_iters) {
    ++t;
    unsigned int changed = 0;
    e = cudaMemset(dchg.p, 0, 4);
    if (e != cudaSuccess) break;
    k_km_assign<<<ablocks, 256>>>((const double *)dF.p, (const double *)dmu.p, n, dim, m, (uint32_t *)dmap.p,
                                  (unsigned int *)dchg.p);
    e = cudaGetLastError();
    if (e == cudaSuccess) e = cudaMemcpy(&changed, dchg.p, 4, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess || changed == 0) break;
    k_km_update<<<ublocks, 256>>>((const double *)dF.p, (const uint32_t *)dmap.p, n, dim, m, (double *)dmu.p);
    e = cudaGetLastError();
    if (e != cudaSuccess) break;
  }
  if (e == cudaSuccess) e = cudaMemcpy(h_map, dmap.p, (size_t)n * 4, cudaMemcpyDeviceToHost);
  if (e == cudaSuccess && h_centroids) e = cudaMemcpy(h_centroids, dmu.p, mu.size() * 8, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return km_fail(NTC_ERR_CUDA, cudaGetErrorString(e));
  if (iters_run) *iters_run = t;
  return NTC_OK;
}
