// Row-pair copy of the latent grids (built once per context).
//
// The gather-decode kernel fetches each bilinear row -- texels (x0, y) and
// (x1, y) of one grid -- with a single 32-byte load.  In the pair copy, texel
// (x, y) of every grid holds [latent(x, y), latent(x1(x), y)], where x1 is the
// right neighbour under the context's address mode: (x + 1) mod W for wrap,
// min(x + 1, W - 1) for clamp.  Grids are laid out back to back in the order
// of their descriptors (pgrids[g].base), so overlapping or gapped placements
// in the caller's latent buffer need no special care.
#include "ntc_internal.cuh"

namespace ntc {
namespace {

__global__ void k_build_pairs(Assets A, const uint32_t *chunk_grid, const uint32_t *chunk_start, uint4 *pair) {
  const uint32_t g = chunk_grid[blockIdx.x], t0 = chunk_start[blockIdx.x];
  const GridDesc src = A.grids[g], dst = A.pgrids[g];
  const uint32_t n = src.W * src.H;
  const uint32_t t1 = min(n, t0 + kPairChunk);
  for (uint32_t t = t0 + threadIdx.x; t < t1; t += blockDim.x) {
    const uint32_t y = t / src.W, x = t - y * src.W;
    uint32_t x1 = x + 1;
    if (x1 == src.W) x1 = A.address_mode == 0 ? 0u : x;
    const uint4 a = A.lat[src.base + t], b = A.lat[src.base + (size_t)y * src.W + x1];
    uint4 *o = pair + 2 * (dst.base + t);
    o[0] = a;
    o[1] = b;
  }
}

}  // namespace

cudaError_t launch_build_pairs(const Assets &A, const uint32_t *chunk_grid, const uint32_t *chunk_start,
                               uint32_t num_chunks, uint4 *pair, cudaStream_t st) {
  if (num_chunks == 0) return cudaSuccess;
  k_build_pairs<<<num_chunks, 256, 0, st>>>(A, chunk_grid, chunk_start, pair);
  return cudaGetLastError();
}

}  // namespace ntc
