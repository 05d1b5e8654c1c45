// Query bucketing: a stable counting sort of the queries by decoder id.
//
// Sec. 2 of the paper defines divergence as several decoders being needed by
// the queries of one block; sorting the queries by decoder (stable, so each
// bucket keeps the original order) turns the interleaved stream into runs of
// single-decoder 128-query tiles.  Two kernels:
//   k_count  the decoder histogram of all queries: per-warp counters in shared
//            memory (one __match_any_sync leader per run of equal decoders),
//            one atomicAdd per decoder and CTA into the global totals
//   k_place  one CTA per 2048-query chunk, chunks taken in ticket order.  It
//            ranks its queries stably within the chunk, publishes its
//            per-decoder counts, and finds how many queries of each decoder
//            the earlier chunks hold by a decoupled look-back over their
//            published counts and inclusive prefixes (it waits only on CTAs
//            that took an earlier ticket, which are already running).  With
//            the segment starts (the scan of the totals) that fixes every
//            query's place; the chunk is sorted in shared memory and copied
//            out with coalesced stores (perm[] and the sorted records).  The
//            CTA with chunk 0 writes the tile table; the last CTA to finish
//            clears the totals and tickets for the next call.
// The permutation is exactly std::stable_sort of the indices by decoder.  A
// query whose set id is out of range goes to the extra bucket D.
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

__device__ __forceinline__ uint64_t globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
constexpr uint64_t kWaitNs = 200ull * 1000ull * 1000ull;  // every wait gives up after 200 ms

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
    const uint64_t now = globaltimer();
    if (spin == 0) t0 = now;
    else if (now - t0 > kWaitNs) return false;
  }
}

// Look-back descriptors, one 64-bit word per (chunk, decoder): the low half is
// a count, the high half (epoch << 2) | state with state 1 = the chunk's own
// count, 2 = the inclusive prefix over chunks 0..c.  A word of another epoch
// (an earlier call) is "not ready", so nothing has to be cleared between calls.
__device__ __forceinline__ unsigned long long ld_desc(const unsigned long long *p) {
  unsigned long long v;
  asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_desc(unsigned long long *p, unsigned long long v) {
  asm volatile("st.relaxed.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ unsigned long long make_desc(uint32_t epoch, uint32_t state, uint32_t count) {
  return ((unsigned long long)((epoch << 2) | state) << 32) | count;
}

// ------------------------------------------------------------------ k_count

__global__ void __launch_bounds__(kBucketThreads) k_count(Assets A, const ntc_query *q, size_t n,
                                                          uint32_t chunks, uint32_t *totals) {
  extern __shared__ uint32_t cnt[];  // [kWarps][D+1]
  pdl_trigger();                     // k_place may start its own work at once
  const uint32_t D1 = A.num_decoders + 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (uint32_t i = threadIdx.x; i < kWarps * D1; i += blockDim.x) cnt[i] = 0;
  __syncthreads();
  const MapLookup lookup(A);
  uint32_t *my = cnt + warp * D1;
  const uint32_t *sid = reinterpret_cast<const uint32_t *>(q);
  for (uint32_t c = blockIdx.x; c < chunks; c += gridDim.x) {
    const size_t wbase = (size_t)c * kBucketChunk + (size_t)warp * (kBucketItems * 32);
    uint32_t s[kBucketItems];
#pragma unroll
    for (int it = 0; it < kBucketItems; ++it) {  // every load in flight before any is used
      const size_t j = wbase + it * 32 + lane;
      s[it] = j < n ? __ldg(sid + 4 * j) : 0u;
    }
#pragma unroll
    for (int it = 0; it < kBucketItems; ++it) {
      const size_t j = wbase + it * 32 + lane;
      const uint32_t dl = lookup(A, s[it]);  // every lane: the lookup shuffles
      const uint32_t d = j < n ? dl : 0xFFFFFFFFu;
      const uint32_t m = __match_any_sync(0xFFFFFFFFu, d);
      if (d != 0xFFFFFFFFu && lane == __ffs(m) - 1) my[d] += __popc(m);
      __syncwarp();
    }
  }
  __syncthreads();
  for (uint32_t d = threadIdx.x; d < D1; d += blockDim.x) {
    uint32_t s = 0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) s += cnt[w * D1 + d];
    if (s) atomicAdd(totals + d, s);
  }
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

// ------------------------------------------------------------------ k_place

// meta layout: [0] num_tiles, [1 .. D+2] seg_start, [D+3 .. 2D+4] tile_start;
// then totals [D+1], the start ticket and the done ticket (zero between calls).
__global__ void __launch_bounds__(kBucketThreads) k_place(Assets A, const ntc_query *q, size_t n,
                                                          uint32_t chunks, uint32_t *meta,
                                                          unsigned long long *desc, uint32_t epoch,
                                                          uint32_t *perm, ntc_query *sorted,
                                                          unsigned int *status) {
  // shared memory: the chunk's records [chunk] (16 B), the chunk-local index
  // [chunk] (u16) and decoder [chunk] (u16) of every sorted slot, then per-warp
  // counters [kWarps][D+1] (reused for the segment starts once the chunk is
  // sorted), and per decoder the chunk-local run start and the global base
  extern __shared__ uint4 srec[];
  __shared__ uint64_t bar;
  __shared__ uint32_t s_chunk;
  __shared__ bool s_last;
  uint16_t *sidx = reinterpret_cast<uint16_t *>(srec + kBucketChunk);
  uint16_t *sdec = sidx + kBucketChunk;
  uint32_t *cnt = reinterpret_cast<uint32_t *>(sdec + kBucketChunk);
  const uint32_t D = A.num_decoders, D1 = D + 1;
  uint32_t *loff = cnt + kWarps * D1;  // chunk-local start of each decoder's run
  uint32_t *gbase = loff + D1;         // global position of that run's first element
  uint32_t *totals = meta + meta_words(D);
  uint32_t *start_ticket = totals + D1, *done_ticket = start_ticket + 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) s_chunk = atomicAdd(start_ticket, 1u);  // chunks in the order CTAs start
  for (uint32_t i = threadIdx.x; i < kWarps * D1; i += blockDim.x) cnt[i] = 0;
  __syncthreads();
  const uint32_t c = s_chunk;
  const size_t cbase = (size_t)c * kBucketChunk;
  const uint32_t valid = (uint32_t)min((size_t)kBucketChunk, n - cbase);
  bulk_issue(srec, q + cbase, valid * 16u, &bar);
  pdl_trigger();  // the decode may launch (it waits for this grid before reading)
  const MapLookup lookup(A);
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
  // per decoder: warp prefix (in place) and the chunk's count, published at
  // once so later chunks can look back past this one
  for (uint32_t d = threadIdx.x; d < D1; d += blockDim.x) {
    uint32_t run = 0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      const uint32_t x = cnt[w * D1 + d];
      cnt[w * D1 + d] = run;
      run += x;
    }
    loff[d] = run;
    gbase[d] = run;  // the count, until the look-back replaces it
    st_desc(desc + (size_t)c * D1 + d, make_desc(epoch, c == 0 ? 2u : 1u, run));
  }
  __syncthreads();
  block_scan_256(loff, D1);  // exclusive scan of the chunk's counts over decoders
  // stable local sort of (local index, decoder) pairs
#pragma unroll
  for (int it = 0; it < kBucketItems; ++it) {
    const uint32_t d = dec[it];
    if (d == 0xFFFFFFFFu) continue;
    const uint32_t lp = loff[d] + cnt[warp * D1 + d] + rank[it];
    sidx[lp] = (uint16_t)(wbase + it * 32 + lane);
    sdec[lp] = (uint16_t)d;
  }
  // decoupled look-back: the queries of decoder d in chunks 0..c-1
  bool gave_up = false;
  for (uint32_t d = threadIdx.x; d < D1; d += blockDim.x) {
    const uint32_t own = gbase[d];
    uint32_t before = 0;
    if (c > 0) {
      uint32_t p = c - 1;
      uint64_t t0 = 0;
      for (uint32_t spin = 0;;) {
        const unsigned long long v = ld_desc(desc + (size_t)p * D1 + d);
        const uint32_t hi = (uint32_t)(v >> 32);
        if ((hi >> 2) == epoch && (hi & 3u) != 0u) {
          before += (uint32_t)v;
          if ((hi & 3u) == 2u || p == 0) break;
          --p;
          continue;
        }
        const uint64_t now = globaltimer();  // chunk p has not published yet
        if (spin++ == 0) t0 = now;
        else if (now - t0 > kWaitNs) {
          gave_up = true;
          break;
        }
      }
      st_desc(desc + (size_t)c * D1 + d, make_desc(epoch, 2u, before + own));
    }
    gbase[d] = before;
  }
  if (gave_up) atomicOr(status, 4u);
  // the totals of k_count give the segment starts (into cnt, free now)
  pdl_wait();
  __syncthreads();
  uint32_t *seg = cnt;
  for (uint32_t d = threadIdx.x; d < D1; d += blockDim.x) seg[d] = __ldcg(totals + d);
  __syncthreads();
  block_scan_256(seg, D1);
  for (uint32_t d = threadIdx.x; d < D1; d += blockDim.x) gbase[d] += seg[d];
  if (c == 0) {  // the tile table: segment starts and tile starts over the D+1 buckets
    uint32_t *mseg = meta + 1, *tst = meta + 1 + (D + 2);
    uint32_t *tiles = seg + D1;  // cnt has kWarps * D1 words
    for (uint32_t d = threadIdx.x; d < D1; d += blockDim.x) {
      mseg[d] = seg[d];
      tiles[d] = (__ldcg(totals + d) + kTile - 1) / kTile;
    }
    __syncthreads();
    const uint32_t last_tiles = tiles[D];
    __syncthreads();
    block_scan_256(tiles, D1);
    for (uint32_t d = threadIdx.x; d < D1; d += blockDim.x) tst[d] = tiles[d];
    if (threadIdx.x == 0) {
      mseg[D1] = (uint32_t)n;
      tst[D1] = tiles[D] + last_tiles;
      meta[0] = tiles[D] + last_tiles;
    }
  }
  __syncthreads();
  // coalesced copy-out: consecutive slots of one decoder go to consecutive
  // positions of that decoder's segment
  for (uint32_t i = threadIdx.x; i < valid; i += blockDim.x) {
    const uint32_t d = sdec[i], j = sidx[i];
    const uint32_t pos = gbase[d] + (i - loff[d]);
    perm[pos] = (uint32_t)(cbase + j);
    reinterpret_cast<uint4 *>(sorted)[pos] = srec[j];
  }
  // the last CTA to finish clears the totals and tickets for the next call
  // (every CTA has read the totals before it takes its done ticket)
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    s_last = atomicAdd(done_ticket, 1u) == chunks - 1;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  for (uint32_t d = threadIdx.x; d < D1; d += blockDim.x) totals[d] = 0;
  if (threadIdx.x == 0) {
    *start_ticket = 0;
    *done_ticket = 0;
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

size_t bucket_chunks(size_t n) { return (n + kBucketChunk - 1) / kBucketChunk; }
size_t bucket_desc_words(uint32_t D, size_t n) { return ((size_t)D + 1) * bucket_chunks(n); }
size_t bucket_meta_words(uint32_t D) { return meta_words(D) + ((size_t)D + 1) + 2; }

cudaError_t launch_bucket(const Assets &A, const ntc_query *q, size_t n, const Scratch &s,
                          cudaStream_t st, int *launches, unsigned int *status) {
  const uint32_t chunks = (uint32_t)bucket_chunks(n);
  const uint32_t D1 = A.num_decoders + 1;
  const size_t smem_count = (size_t)kWarps * D1 * sizeof(uint32_t);
  const size_t smem_place = (size_t)kBucketChunk * (16 + 2 + 2) + (size_t)(kWarps + 2) * D1 * sizeof(uint32_t);
  static PerDevice attrs;
  cudaError_t e = attrs.once([]() {
    cudaError_t r = cudaFuncSetAttribute(k_count, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
    if (r == cudaSuccess)
      r = cudaFuncSetAttribute(k_place, cudaFuncAttributeMaxDynamicSharedMemorySize, 210 * 1024);
    return r;
  });
  if (e != cudaSuccess) return e;
  int dev = 0, sms = 1, smem_sm = 233472, thr_sm = 2048;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cudaDeviceGetAttribute(&smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev);
  cudaDeviceGetAttribute(&thr_sm, cudaDevAttrMaxThreadsPerMultiProcessor, dev);
  // k_count: a grid that is resident at once (by threads and by its shared
  // memory, which grows with the decoder count), each CTA striding over chunks
  size_t occ = (size_t)thr_sm / kBucketThreads;
  const size_t by_smem = (size_t)smem_sm / (smem_count + 1024);
  if (by_smem < occ) occ = by_smem;
  if (occ < 1) occ = 1;
  size_t grid = (size_t)sms * occ;
  if (grid > chunks) grid = chunks;
  uint32_t *totals = s.meta + meta_words(A.num_decoders);
  k_count<<<(unsigned)grid, kBucketThreads, smem_count, st>>>(A, q, n, chunks, totals);
  e = launch_pdl(k_place, dim3(chunks), dim3(kBucketThreads), smem_place, st, A, q, n, chunks, s.meta, s.desc,
                 s.epoch, s.perm, s.sorted, status);
  *launches += 2;
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
