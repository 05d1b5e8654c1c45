// Query bucketing: a stable counting sort of the queries by decoder id.
//
// Sec. 2 of the paper defines divergence as several decoders being needed by
// the queries of one block; sorting the queries by decoder (stable, so each
// bucket keeps the original order) turns the interleaved stream into runs of
// single-decoder 128-query tiles.  Three kernels, no inter-CTA waiting:
//   k_hist    per-chunk histogram; each warp of a chunk owns a contiguous range
//             and counts it with __match_any_sync (one leader per decoder run)
//   k_scan    one CTA per decoder scans that decoder's per-chunk counts; the last
//             CTA to finish (atomic ticket) scans the decoder totals into the
//             segment starts and the tile starts
//   k_scatter recomputes each warp's counts, sorts its chunk stably by decoder
//             in shared memory, then copies each decoder's run out to its
//             segment with coalesced stores (perm[] and the sorted records)
// A query whose set id is out of range goes to the extra bucket D.
#include "ntc_internal.cuh"

namespace ntc {
namespace {

constexpr int kWarps = kBucketThreads / 32;

__device__ __forceinline__ uint32_t decoder_of(const Assets &A, uint32_t set_id) {
  return set_id < A.num_sets ? __ldg(A.map + set_id) : A.num_decoders;
}

// The set -> decoder map of up to 32 sets lives in one register per lane
// (lane s holds map[s]); larger maps are read through the cache.
struct MapLookup {
  uint32_t reg;
  bool small;
  __device__ explicit MapLookup(const Assets &A) {
    const uint32_t lane = threadIdx.x & 31;
    small = A.num_sets <= 32;
    reg = small && lane < A.num_sets ? __ldg(A.map + lane) : A.num_decoders;
  }
  // called by all 32 lanes of the warp together
  __device__ __forceinline__ uint32_t operator()(const Assets &A, uint32_t set_id) const {
    if (small) {
      const uint32_t d = __shfl_sync(0xFFFFFFFFu, reg, set_id & 31);
      return set_id < A.num_sets ? d : A.num_decoders;
    }
    return decoder_of(A, set_id);
  }
};

__device__ __forceinline__ uint32_t saddr_b(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

// Stream `bytes` (a multiple of 16) from global memory into shared memory with
// one bulk copy (TMA): bulk_issue (every thread; thread 0 issues), then
// bulk_wait, which is false if the copy has not landed after 200 ms.
__device__ void bulk_issue(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
  const uint32_t b = saddr_b(bar);
  if (threadIdx.x == 0) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;\n" ::"r"(b) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(b), "r"(bytes) : "memory");
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];\n" ::"r"(
                     saddr_b(dst)),
                 "l"(src), "r"(bytes), "r"(b)
                 : "memory");
  }
  __syncthreads();
}

__device__ bool bulk_wait(uint64_t *bar) {
  const uint32_t b = saddr_b(bar);
  uint64_t t0 = 0;
  for (uint32_t spin = 0;; ++spin) {
    uint32_t ok;
    asm volatile(
        "{\n.reg .pred p;\nmbarrier.try_wait.parity.shared::cta.b64 p, [%1], 0;\nselp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(b)
        : "memory");
    if (ok) return true;
    uint64_t now;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(now));
    if (spin == 0) t0 = now;
    else if (now - t0 > 200ull * 1000ull * 1000ull) return false;
  }
}

__global__ void __launch_bounds__(kBucketThreads) k_hist(Assets A, const ntc_query *q, size_t n,
                                                         uint32_t *counts, uint32_t chunks,
                                                         unsigned int *status) {
  // shared memory: the chunk's records [kBucketChunk], then [kWarps][D+1] counters
  extern __shared__ uint4 srec[];
  __shared__ uint64_t bar;
  uint32_t *cnt = reinterpret_cast<uint32_t *>(srec + kBucketChunk);
  const uint32_t D1 = A.num_decoders + 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const MapLookup lookup(A);
  const size_t cbase = (size_t)blockIdx.x * kBucketChunk;
  const uint32_t valid = (uint32_t)min((size_t)kBucketChunk, n - cbase);
  for (uint32_t i = threadIdx.x; i < kWarps * D1; i += blockDim.x) cnt[i] = 0;
  bulk_issue(srec, q + cbase, valid * 16u, &bar);
  pdl_trigger();  // k_scan may launch (it waits for this grid before reading)
  if (!bulk_wait(&bar)) atomicOr(status, 2u);
  const uint32_t wbase = (uint32_t)warp * (kBucketItems * 32);
  uint32_t *my = cnt + warp * D1;
#pragma unroll
  for (int it = 0; it < kBucketItems; ++it) {
    const uint32_t j = wbase + it * 32 + lane;
    const uint32_t dl = lookup(A, j < valid ? srec[j].x : 0u);  // every lane: the lookup shuffles
    const uint32_t d = j < valid ? dl : 0xFFFFFFFFu;
    const uint32_t m = __match_any_sync(0xFFFFFFFFu, d);
    if (d != 0xFFFFFFFFu && lane == __ffs(m) - 1) my[d] += __popc(m);
    __syncwarp();
  }
  __syncthreads();
  for (uint32_t d = threadIdx.x; d < D1; d += blockDim.x) {
    uint32_t s = 0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) s += cnt[w * D1 + d];
    counts[(size_t)d * chunks + blockIdx.x] = s;
  }
}

// Exclusive scan of one value per thread over a 1024-thread block.
__device__ __forceinline__ uint32_t block_scan_1024(uint32_t v, uint32_t &total, uint32_t *ws) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    uint32_t y = __shfl_up_sync(0xFFFFFFFFu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) ws[warp] = x;
  __syncthreads();
  if (warp == 0) {
    uint32_t s = ws[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      uint32_t y = __shfl_up_sync(0xFFFFFFFFu, s, o);
      if (lane >= o) s += y;
    }
    ws[lane] = s;
  }
  __syncthreads();
  uint32_t excl = x - v + (warp > 0 ? ws[warp - 1] : 0u);
  total = ws[31];
  __syncthreads();
  return excl;
}

// Scan `len` values in place (exclusive) with 1024 threads, 4 per thread per
// round; returns the total.
__device__ uint32_t block_scan_inplace(uint32_t *a, uint32_t len, uint32_t *ws) {
  uint32_t carry = 0;
  for (uint32_t b = 0; b < len; b += 4096) {
    uint32_t v[4], s = 0;
    const uint32_t i0 = b + threadIdx.x * 4;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      v[j] = i0 + j < len ? a[i0 + j] : 0u;
      s += v[j];
    }
    uint32_t tot;
    uint32_t e = block_scan_1024(s, tot, ws) + carry;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      if (i0 + j < len) a[i0 + j] = e;
      e += v[j];
    }
    carry += tot;
  }
  return carry;
}

// meta layout: [0] num_tiles, [1 .. D+2] seg_start, [D+3 .. 2D+4] tile_start;
// ticket: one word, zero between calls.
__global__ void __launch_bounds__(1024) k_scan(uint32_t *counts, uint32_t chunks, uint32_t D,
                                               uint32_t n, uint32_t *totals, uint32_t *meta,
                                               uint32_t *ticket) {
  __shared__ uint32_t ws[32];
  __shared__ bool last;
  const uint32_t d = blockIdx.x;
  pdl_wait();  // the per-chunk counts of k_hist
  uint32_t tot = block_scan_inplace(counts + (size_t)d * chunks, chunks, ws);
  if (threadIdx.x == 0) {
    totals[d] = tot;
    __threadfence();
    last = atomicAdd(ticket, 1u) == D;  // gridDim.x == D + 1
  }
  __syncthreads();
  if (!last) return;
  __threadfence();
  uint32_t *seg = meta + 1, *tst = meta + 1 + (D + 2);
  // segment starts and tile starts over the D+1 buckets
  for (uint32_t i = threadIdx.x; i < D + 1; i += blockDim.x) {
    uint32_t c = ((volatile uint32_t *)totals)[i];
    seg[i] = c;
    tst[i] = (c + kTile - 1) / kTile;
  }
  __syncthreads();
  uint32_t ns = block_scan_inplace(seg, D + 1, ws);
  __syncthreads();
  uint32_t nt = block_scan_inplace(tst, D + 1, ws);
  if (threadIdx.x == 0) {
    seg[D + 1] = ns;  // == n
    tst[D + 1] = nt;
    meta[0] = nt;
    *ticket = 0;
  }
  (void)n;
}

// In-place exclusive scan of len values (in shared memory) by the 256 threads of
// a block, each over a contiguous run of ceil(len / 256) values.
__device__ void block_scan_256(uint32_t *a, uint32_t len) {
  __shared__ uint32_t wsum[kWarps];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t per = (len + kBucketThreads - 1) / kBucketThreads;
  const uint32_t b = threadIdx.x * per, e = min(len, b + per);
  uint32_t s = 0;
  for (uint32_t i = b; i < e; ++i) s += a[i];
  uint32_t x = s;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) wsum[warp] = x;
  __syncthreads();
  uint32_t wp = 0;
  for (int w = 0; w < warp; ++w) wp += wsum[w];
  uint32_t run = wp + x - s;
  for (uint32_t i = b; i < e; ++i) {
    const uint32_t c = a[i];
    a[i] = run;
    run += c;
  }
  __syncthreads();
}

// SPREAD (the single-pass bucketing of the tensor-core decode): no k_hist or
// k_scan runs first.  Decoder d owns region [d * cap, d * cap + cap) of perm
// and sorted (cap = n); each chunk reserves room for its run of decoder d with
// one atomicAdd on cursor[d], so runs of one decoder keep chunk order only as
// far as the atomics happen to, and the permutation is not the stable one
// (every decoded row is independent of the others in its tile, so outputs do
// not change).  The last CTA to finish (atomic ticket, no waiting) writes meta
// with seg[d] = the decoder's count and the tile starts, and clears cursor and
// ticket for the next call.
template <bool SPREAD>
__global__ void __launch_bounds__(kBucketThreads) k_scatter(Assets A, const ntc_query *q, size_t n,
                                                            const uint32_t *counts, uint32_t chunks,
                                                            uint32_t *meta, uint32_t *perm,
                                                            ntc_query *sorted, unsigned int *status,
                                                            uint32_t *cursor, uint32_t cap) {
  // shared memory: the chunk's records [chunk] (16 B), the chunk-local index
  // [chunk] (u16) and decoder [chunk] (u16) of every sorted slot, then per-warp
  // counters [kWarps][D+1] and the chunk's per-decoder local offsets and global
  // bases [D+1] each
  extern __shared__ uint4 srec[];
  __shared__ uint64_t bar;
  uint16_t *sidx = reinterpret_cast<uint16_t *>(srec + kBucketChunk);
  uint16_t *sdec = sidx + kBucketChunk;
  uint32_t *cnt = reinterpret_cast<uint32_t *>(sdec + kBucketChunk);
  const uint32_t D1 = A.num_decoders + 1;
  uint32_t *loff = cnt + kWarps * D1;  // chunk-local start of each decoder's run
  uint32_t *gbase = loff + D1;         // global position of that run's first element
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const MapLookup lookup(A);
  const size_t cbase = (size_t)blockIdx.x * kBucketChunk;
  const uint32_t valid = (uint32_t)min((size_t)kBucketChunk, n - cbase);
  for (uint32_t i = threadIdx.x; i < kWarps * D1; i += blockDim.x) cnt[i] = 0;
  bulk_issue(srec, q + cbase, valid * 16u, &bar);  // the queries do not depend on k_scan
  if (!SPREAD) pdl_wait();                           // the scanned counts and segment starts
  pdl_trigger();                                     // the decode may launch (it waits for this grid)
  if (!bulk_wait(&bar)) atomicOr(status, 2u);
  const uint32_t wbase = (uint32_t)warp * (kBucketItems * 32);  // this warp's run in the chunk
  uint32_t dec[kBucketItems];
#pragma unroll
  for (int it = 0; it < kBucketItems; ++it) {
    const uint32_t j = wbase + it * 32 + lane;
    const uint32_t dl = lookup(A, j < valid ? srec[j].x : 0u);  // every lane: the lookup shuffles
    dec[it] = j < valid ? dl : 0xFFFFFFFFu;
  }
  uint32_t *my = cnt + warp * D1;
  // rank of each query among the equal decoders of this warp's run, in order
  uint32_t rank[kBucketItems];
  const uint32_t lt = (1u << lane) - 1u;
#pragma unroll
  for (int it = 0; it < kBucketItems; ++it) {
    const uint32_t d = dec[it];
    const uint32_t m = __match_any_sync(0xFFFFFFFFu, d);
    rank[it] = d != 0xFFFFFFFFu ? my[d] + __popc(m & lt) : 0u;
    __syncwarp();
    if (d != 0xFFFFFFFFu && lane == __ffs(m) - 1) my[d] += __popc(m);
    __syncwarp();
  }
  __syncthreads();
  // per decoder: warp prefix (in place), chunk total and global base.  SPREAD
  // with D + 1 <= blockDim.x: thread d keeps its reservation in a register
  // until the copy-out, so the atomic's round trip overlaps the scan and the
  // local sort
  const uint32_t *seg = meta + 1;
  const bool reg_base = SPREAD && D1 <= blockDim.x;
  uint32_t my_base = 0;
  for (uint32_t d = threadIdx.x; d < D1; d += blockDim.x) {
    uint32_t run = 0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      const uint32_t c = cnt[w * D1 + d];
      cnt[w * D1 + d] = run;
      run += c;
    }
    loff[d] = run;
    if (SPREAD) {
      const uint32_t b = run ? d * cap + atomicAdd(cursor + d, run) : 0u;
      if (reg_base) my_base = b;
      else gbase[d] = b;
    } else {
      gbase[d] = __ldg(seg + d) + counts[(size_t)d * chunks + blockIdx.x];
    }
  }
  __syncthreads();
  block_scan_256(loff, D1);  // exclusive scan of the chunk totals over decoders
  // stable local sort of (local index, decoder) pairs
#pragma unroll
  for (int it = 0; it < kBucketItems; ++it) {
    const uint32_t d = dec[it];
    if (d == 0xFFFFFFFFu) continue;
    const uint32_t lp = loff[d] + cnt[warp * D1 + d] + rank[it];
    sidx[lp] = (uint16_t)(wbase + it * 32 + lane);
    sdec[lp] = (uint16_t)d;
  }
  if (reg_base && threadIdx.x < D1) gbase[threadIdx.x] = my_base;
  __syncthreads();
  // SPREAD: every reservation of this chunk has been made (their results are in
  // gbase), so the chunk takes its ticket now, before thread 0 has any global
  // store in flight; the atomic's round trip overlaps the copy-out
  uint32_t ticket_no = 0;
  if (SPREAD && threadIdx.x == 0) {
    __threadfence();  // this CTA's reservations before its ticket
    ticket_no = atomicAdd(cursor + D1, 1u);
  }
  // coalesced copy-out: consecutive slots of one decoder go to consecutive
  // positions of that decoder's segment
  for (uint32_t i = threadIdx.x; i < valid; i += blockDim.x) {
    const uint32_t d = sdec[i], j = sidx[i];
    const uint32_t pos = gbase[d] + (i - loff[d]);
    perm[pos] = (uint32_t)(cbase + j);
    reinterpret_cast<uint4 *>(sorted)[pos] = srec[j];
  }
  if (SPREAD) {
    __shared__ bool last;
    uint32_t *ticket = cursor + D1;
    if (threadIdx.x == 0) last = ticket_no == gridDim.x - 1;
    __syncthreads();
    if (!last) return;
    __threadfence();
    // every chunk has reserved its runs: counts per decoder and tile starts
    uint32_t *segc = meta + 1, *tst = meta + 1 + (D1 + 1);
    for (uint32_t d = threadIdx.x; d < D1; d += blockDim.x) {
      const uint32_t c = ((volatile uint32_t *)cursor)[d];
      segc[d] = c;
      loff[d] = (c + kTile - 1) / kTile;
      cursor[d] = 0;
    }
    __syncthreads();
    const uint32_t last_tiles = loff[D1 - 1];
    __syncthreads();
    block_scan_256(loff, D1);
    for (uint32_t d = threadIdx.x; d < D1; d += blockDim.x) tst[d] = loff[d];
    if (threadIdx.x == 0) {
      const uint32_t T = loff[D1 - 1] + last_tiles;
      tst[D1] = T;
      segc[D1] = 0;
      meta[0] = T;
      *ticket = 0;
    }
  }
}

__global__ void k_tiles_export(const uint32_t *meta, uint32_t D, uint32_t *tiles, uint32_t *num_tiles,
                               uint32_t *counts, size_t max_tiles) {
  const uint32_t T = meta[0];
  const size_t stride = (size_t)gridDim.x * blockDim.x;
  for (size_t t = (size_t)blockIdx.x * blockDim.x + threadIdx.x; t < max_tiles; t += stride) {
    if (tiles && t < T) {
      uint32_t dec, start, len;
      tile_info(meta, D, (uint32_t)t, dec, start, len);
      tiles[3 * t] = dec;
      tiles[3 * t + 1] = start;
      tiles[3 * t + 2] = len;
    }
    if (counts && t < D + 1) counts[t] = meta[1 + t + 1] - meta[1 + t];
  }
  if (num_tiles && blockIdx.x == 0 && threadIdx.x == 0) *num_tiles = T;
}

}  // namespace

size_t bucket_scratch_counts(uint32_t D, size_t n) {
  size_t chunks = (n + kBucketChunk - 1) / kBucketChunk;
  return (size_t)(D + 1) * chunks;
}

cudaError_t launch_bucket(const Assets &A, const ntc_query *q, size_t n, const Scratch &s,
                          cudaStream_t st, int *launches, unsigned int *status) {
  const uint32_t chunks = (uint32_t)((n + kBucketChunk - 1) / kBucketChunk);
  const uint32_t D = A.num_decoders;
  const size_t cnt_bytes = (size_t)kWarps * (D + 1) * sizeof(uint32_t);
  const size_t smem = (size_t)kBucketChunk * 16 + cnt_bytes;
  const size_t smem_scatter = (size_t)kBucketChunk * (16 + 2 + 2) + cnt_bytes + 2 * (D + 1) * sizeof(uint32_t);
  static bool attr_done = false;
  if (!attr_done) {
    cudaFuncSetAttribute(k_hist, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
    cudaFuncSetAttribute(k_scatter<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
    attr_done = true;
  }
  // totals[D+1] and the ticket live after meta
  uint32_t *totals = s.meta + meta_words(D);
  uint32_t *ticket = totals + (D + 1);
  if (s.cursor) {  // single pass: reserve runs in per-decoder regions
    cudaFuncSetAttribute(k_scatter<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
    k_scatter<true><<<chunks, kBucketThreads, smem_scatter, st>>>(A, q, n, nullptr, chunks, s.meta, s.perm,
                                                                   s.sorted, status, s.cursor, s.cap);
    *launches += 1;
    return cudaGetLastError();
  }
  k_hist<<<chunks, kBucketThreads, smem, st>>>(A, q, n, s.counts, chunks, status);
  cudaError_t e = launch_pdl(k_scan, dim3(D + 1), dim3(1024), 0, st, s.counts, chunks, D, (uint32_t)n, totals,
                             s.meta, ticket);
  if (e == cudaSuccess)
    e = launch_pdl(k_scatter<false>, dim3(chunks), dim3(kBucketThreads), smem_scatter, st, A, q, n,
                   (const uint32_t *)s.counts, chunks, s.meta, s.perm, s.sorted, status, (uint32_t *)nullptr,
                   0u);
  *launches += 3;
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

cudaError_t launch_tiles_export(const uint32_t *meta, uint32_t D, uint32_t *tiles, uint32_t *num_tiles,
                                uint32_t *counts, size_t max_tiles, cudaStream_t st, int *launches) {
  size_t work = max_tiles > (size_t)D + 1 ? max_tiles : (size_t)D + 1;
  unsigned blocks = (unsigned)((work + 255) / 256);
  if (blocks > 4096) blocks = 4096;
  k_tiles_export<<<blocks, 256, 0, st>>>(meta, D, tiles, num_tiles, counts, work);
  *launches += 1;
  return cudaGetLastError();
}

}  // namespace ntc
