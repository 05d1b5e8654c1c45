// Query bucketing: a stable counting sort of the queries by decoder id.
//
// Sec. 2 of the paper defines divergence as several decoders being needed by
// the queries of one block; sorting the queries by decoder (stable, so each
// bucket keeps the original order) turns the interleaved stream into runs of
// single-decoder 128-query tiles.  Three kernels, none of which waits for
// another CTA:
//   k_count  per 2048-query chunk: every query's decoder (set -> decoder map;
//            out-of-range set ids form the extra bucket D), written as one
//            byte (two beyond 255 decoders), the chunk's count of every
//            decoder, and the divergence of its 32-query groups (Eq. 1:
//            distinct decoders in a group - 1, summed)
//   k_scan   one CTA per decoder scans that decoder's per-chunk counts into
//            the chunk offsets (an array of their own: the counts are only
//            read, so the kernel can run again on them, as a profiler's
//            replay does); the last CTA to finish (atomic ticket) scans
//            the decoder totals into the segment starts and the tile starts,
//            and decides from Eq. 1's score whether the records are copied
//   k_place  per chunk: each query's rank among the equal decoders of its
//            chunk (stable); its place = segment start + chunk offset + rank.
//            When k_scan chose to copy the records, the chunk is sorted in
//            shared memory and copied out with coalesced stores: perm[] and
//            the query records in bucket order (staged by cp.async).
//            Otherwise each perm entry is stored straight to its place: the
//            equal decoders of a 32-query group get consecutive places, so a
//            single-decoder group's stores coalesce
// Divergence-aware: when the score is low (a G-buffer: most 32-query groups
// need one decoder) a decoder's queries lie in long runs of the caller's
// array, and the decode reads query perm[i] there directly; only a scattered
// stream (score above kCopyAboveScore) pays for the copy, so its decode reads
// contiguous records.  Equal decoders within a warp are found with one ballot
// per bit of the decoder id.  The permutation is exactly std::stable_sort of
// the indices by decoder.
#include <algorithm>

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

// Bits that hold every key of a call: the buckets 0..D plus D + 1 for "no
// query" (a lane past the end).
__device__ __forceinline__ int key_bits(uint32_t D) { return 32 - __clz(D + 1); }

// The lanes of the warp whose key equals this lane's: one ballot per key bit
// (each lane keeps the lanes that agree with it on that bit), after a check
// for the common case of a G-buffer, one key in the whole warp.
__device__ __forceinline__ uint32_t match_key(uint32_t key, int nbits) {
  if (__all_sync(0xFFFFFFFFu, key == __shfl_sync(0xFFFFFFFFu, key, 0))) return 0xFFFFFFFFu;
  uint32_t m = 0xFFFFFFFFu;
  for (int b = 0; b < nbits; ++b) {
    const bool bit = (key >> b) & 1u;
    const uint32_t bal = __ballot_sync(0xFFFFFFFFu, bit);
    m &= bit ? bal : ~bal;
  }
  return m;
}

// ------------------------------------------------------------------ k_count

template <typename DecT>
__global__ void __launch_bounds__(kBucketThreads) k_count(Assets A, const ntc_query *q, size_t n,
                                                             uint32_t chunks, uint32_t *counts, uint32_t *div_sum,
                                                             DecT *dec_out) {
  extern __shared__ uint32_t cnt[];  // [kWarps][D+2]; column D+1 counts nothing
  __shared__ uint32_t s_div;
  pdl_trigger();                     // k_scan may launch (it waits for this grid before reading)
  const uint32_t D = A.num_decoders, DW = D + 2;
  if (threadIdx.x == 0) s_div = 0;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (uint32_t i = threadIdx.x; i < kWarps * DW; i += blockDim.x) cnt[i] = 0;
  __syncthreads();
  const MapLookup lookup(A);
  const int nbits = key_bits(D);
  const size_t wbase = (size_t)blockIdx.x * kBucketChunk + (size_t)warp * (kBucketItems * 32);
  const uint32_t *sid = reinterpret_cast<const uint32_t *>(q);
  uint32_t s[kBucketItems];
#pragma unroll
  for (int it = 0; it < kBucketItems; ++it) {  // every load in flight before any is used
    const size_t j = wbase + it * 32 + lane;
    s[it] = j < n ? __ldg(sid + 4 * j) : 0u;
  }
  uint32_t *my = cnt + warp * DW;
  uint32_t div = 0;  // this warp's groups: distinct decoders - 1
  uint32_t dv[kBucketItems];
#pragma unroll
  for (int it = 0; it < kBucketItems; ++it) {
    const size_t j = wbase + it * 32 + lane;
    const uint32_t dl = lookup(A, s[it]);  // every lane: the lookup shuffles
    dv[it] = j < n ? dl : D + 1;
    if (dec_out && j < n) dec_out[j] = (DecT)dv[it];
  }
  // a warp whose 256 queries all need one decoder (most of a G-buffer's):
  // one count, no divergence
  const uint32_t d0 = __shfl_sync(0xFFFFFFFFu, dv[0], 0);
  bool one = true;
#pragma unroll
  for (int it = 0; it < kBucketItems; ++it) one &= dv[it] == d0;
  if (__all_sync(0xFFFFFFFFu, one)) {
    if (lane == 0) my[d0] += kBucketItems * 32;
  } else {
#pragma unroll
    for (int it = 0; it < kBucketItems; ++it) {
      const uint32_t d = dv[it];
      const uint32_t m = match_key(d, nbits);
      const bool leader = lane == __ffs(m) - 1;
      if (leader) my[d] += __popc(m);
      const uint32_t runs = __popc(__ballot_sync(0xFFFFFFFFu, leader && d <= D));
      div += runs ? runs - 1 : 0u;
      __syncwarp();
    }
  }
  if (lane == 0 && div) atomicAdd(&s_div, div);
  __syncthreads();
  if (threadIdx.x == 0 && s_div) atomicAdd(div_sum, s_div);
  for (uint32_t d = threadIdx.x; d <= D; d += blockDim.x) {
    uint32_t t = 0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) t += cnt[w * DW + d];
    counts[(size_t)d * chunks + blockIdx.x] = t;
  }
}

// ------------------------------------------------------------------- k_scan

// Exclusive scan of one value per thread over a 1024-thread block.
__device__ __forceinline__ uint32_t block_scan_1024(uint32_t v, uint32_t &total, uint32_t *ws) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) ws[warp] = x;
  __syncthreads();
  if (warp == 0) {
    uint32_t s = ws[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, s, o);
      if (lane >= o) s += y;
    }
    ws[lane] = s;
  }
  __syncthreads();
  const uint32_t excl = x - v + (warp > 0 ? ws[warp - 1] : 0u);
  total = ws[31];
  __syncthreads();
  return excl;
}

// Exclusive scan of `len` values of src into dst (dst may be src) with 1024
// threads, 4 per thread per round; returns the total.
__device__ uint32_t block_scan_to(const uint32_t *src, uint32_t *dst, uint32_t len, uint32_t *ws) {
  uint32_t carry = 0;
  for (uint32_t b = 0; b < len; b += 4096) {
    uint32_t v[4], s = 0;
    const uint32_t i0 = b + threadIdx.x * 4;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      v[j] = i0 + j < len ? src[i0 + j] : 0u;
      s += v[j];
    }
    uint32_t tot;
    uint32_t e = block_scan_1024(s, tot, ws) + carry;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      if (i0 + j < len) dst[i0 + j] = e;
      e += v[j];
    }
    carry += tot;
  }
  return carry;
}

// meta layout: [0] num_tiles, [1 .. D+2] seg_start, [D+3 .. 2D+4] tile_start,
// [2D+5] copied, [2D+6] divergence; then totals [D+1], the ticket and the
// divergence sum of k_count (zero between calls).
__global__ void __launch_bounds__(1024) k_scan(const uint32_t *counts, uint32_t *offs, uint32_t chunks, uint32_t D,
                                               uint32_t *meta, int force_copy) {
  __shared__ uint32_t ws[32];
  __shared__ bool last;
  const uint32_t d = blockIdx.x;
  uint32_t *totals = meta + meta_words(D), *ticket = totals + (D + 1), *div_sum = ticket + 1;
  pdl_wait();     // the per-chunk counts of k_count
  pdl_trigger();  // k_place may launch (it waits for this grid before reading)
  const uint32_t tot = block_scan_to(counts + (size_t)d * chunks, offs + (size_t)d * chunks, chunks, ws);
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
    const uint32_t c = ((volatile uint32_t *)totals)[i];
    seg[i] = c;
    tst[i] = (c + kTile - 1) / kTile;
  }
  __syncthreads();
  const uint32_t ns = block_scan_to(seg, seg, D + 1, ws);
  __syncthreads();
  const uint32_t nt = block_scan_to(tst, tst, D + 1, ws);
  if (threadIdx.x == 0) {
    seg[D + 1] = ns;  // == n
    tst[D + 1] = nt;
    meta[0] = nt;
    // Eq. 1's score: divergence sum over the ceil(n / 32) groups
    const uint32_t div = *(volatile uint32_t *)div_sum;
    const uint64_t groups = ((uint64_t)ns + 31) / 32;
    meta[meta_copied(D)] = force_copy || (uint64_t)div > (uint64_t)kCopyAboveScore * groups ? 1u : 0u;
    meta[meta_divergence(D)] = div;
    *div_sum = 0;
    *ticket = 0;
  }
}

// ------------------------------------------------------------------ k_place

// In-place exclusive scan of len values (in shared memory) by the threads of a
// block, each over a contiguous run of ceil(len / kBucketThreads) values.
__device__ void block_scan(uint32_t *a, uint32_t len) {
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

__device__ __forceinline__ void cp_async16(void *smem_dst, const void *src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"((uint32_t)__cvta_generic_to_shared(smem_dst)),
               "l"(src)
               : "memory");
}

// FROM_Q: the decoders come from the staged records (always copied);
// otherwise from k_count's decoder array, and the records are staged only
// when k_scan chose to copy them.  A resident grid: each CTA takes chunks
// blockIdx.x, + gridDim.x, ... and loads the next chunk's decoders and chunk
// offsets while it ranks and places the current one.
template <typename DecT, bool FROM_Q>
__global__ void __launch_bounds__(kBucketThreads, 5) k_place(Assets A, const ntc_query *q, const DecT *dec_in,
                                                             size_t n, uint32_t chunks, const uint32_t *offs,
                                                             const uint32_t *meta, uint32_t *perm,
                                                             ntc_query *sorted) {
  // shared memory: the chunk's records [chunk] (16 B), the chunk-local index
  // and decoder of every sorted slot [chunk] (u16 each), per-warp counters
  // [kWarps][D+2], and per decoder the chunk-local run start, the global base
  // and the segment start [D+2] each
  extern __shared__ uint4 srec[];
  uint16_t *sidx = reinterpret_cast<uint16_t *>(srec + kBucketChunk);
  uint16_t *sdec = sidx + kBucketChunk;
  uint32_t *cnt = reinterpret_cast<uint32_t *>(sdec + kBucketChunk);
  const uint32_t D = A.num_decoders, DW = D + 2;
  uint32_t *loff = cnt + kWarps * DW;
  uint32_t *gbase = loff + DW;
  uint32_t *sseg = gbase + DW;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t wbase = (uint32_t)warp * (kBucketItems * 32);  // this warp's run in a chunk
  const uint32_t lt = (1u << lane) - 1u;
  const bool own_offset = D + 1 <= (uint32_t)blockDim.x;       // thread d prefetches decoder d's offset
  auto stage_records = [&](size_t cbase, uint32_t valid) {
    for (uint32_t i = threadIdx.x; i < valid; i += blockDim.x) cp_async16(srec + i, q + cbase + i);
    asm volatile("cp.async.commit_group;\n" ::: "memory");
  };
  auto load_decoders = [&](uint32_t c, uint32_t (&d)[kBucketItems]) {
    const size_t cbase = (size_t)c * kBucketChunk;
    const uint32_t valid = (uint32_t)min((size_t)kBucketChunk, n - cbase);
#pragma unroll
    for (int it = 0; it < kBucketItems; ++it) {
      const uint32_t j = wbase + it * 32 + lane;
      d[it] = j < valid ? (uint32_t)__ldcg(dec_in + cbase + j) : D + 1;
    }
  };
  uint32_t c = blockIdx.x;
  if (FROM_Q && c < chunks)  // the caller's queries: no dependence on k_scan
    stage_records((size_t)c * kBucketChunk, (uint32_t)min((size_t)kBucketChunk, n - (size_t)c * kBucketChunk));
  for (uint32_t i = threadIdx.x; i < kWarps * DW; i += blockDim.x) cnt[i] = 0;
  const MapLookup lookup(A);
  const int nbits = key_bits(D);
  pdl_wait();  // k_scan's chunk offsets, segment starts and decision (and k_count's decoders)
  const bool copy = FROM_Q || __ldcg(meta + meta_copied(D)) != 0u;
  for (uint32_t d = threadIdx.x; d <= D; d += blockDim.x) sseg[d] = __ldcg(meta + 1 + d);
  uint32_t next_dec[kBucketItems], next_off = 0;
  if (!FROM_Q && c < chunks) load_decoders(c, next_dec);
  if (own_offset && threadIdx.x <= D && c < chunks) next_off = __ldcg(offs + (size_t)threadIdx.x * chunks + c);
  for (; c < chunks; c += gridDim.x) {
    const size_t cbase = (size_t)c * kBucketChunk;
    const uint32_t valid = (uint32_t)min((size_t)kBucketChunk, n - cbase);
    const bool last = c + gridDim.x >= chunks;
    if (!FROM_Q && copy) stage_records(cbase, valid);
    uint32_t dec[kBucketItems];
    const uint32_t off = next_off;
    if (FROM_Q) {
      asm volatile("cp.async.wait_all;\n" ::: "memory");
      __syncthreads();
#pragma unroll
      for (int it = 0; it < kBucketItems; ++it) {
        const uint32_t j = wbase + it * 32 + lane;
        const uint32_t dl = lookup(A, j < valid ? srec[j].x : 0u);  // every lane: the lookup shuffles
        dec[it] = j < valid ? dl : D + 1;
      }
    } else {
#pragma unroll
      for (int it = 0; it < kBucketItems; ++it) dec[it] = next_dec[it];
      if (!last) load_decoders(c + gridDim.x, next_dec);  // in flight while this chunk is placed
    }
    if (own_offset && threadIdx.x <= D && !last)
      next_off = __ldcg(offs + (size_t)threadIdx.x * chunks + c + gridDim.x);
    // rank of each query among the equal decoders of this warp's run, in
    // order; a warp whose 256 queries all need one decoder ranks them at once
    uint32_t *my = cnt + warp * DW;
    uint32_t rank[kBucketItems];
    const uint32_t d0 = __shfl_sync(0xFFFFFFFFu, dec[0], 0);
    bool one = true;
#pragma unroll
    for (int it = 0; it < kBucketItems; ++it) one &= dec[it] == d0;
    one = __all_sync(0xFFFFFFFFu, one);  // the warp's 256 queries need decoder d0
    if (one) {
#pragma unroll
      for (int it = 0; it < kBucketItems; ++it) rank[it] = it * 32 + lane;  // my[d0] is 0: a fresh chunk
      if (lane == 0) my[d0] = kBucketItems * 32;
      __syncwarp();
    } else {
#pragma unroll
      for (int it = 0; it < kBucketItems; ++it) {
        const uint32_t d = dec[it];
        const uint32_t m = match_key(d, nbits);
        rank[it] = my[d] + __popc(m & lt);
        __syncwarp();
        if (lane == __ffs(m) - 1) my[d] += __popc(m);
        __syncwarp();
      }
    }
    __syncthreads();
    // per decoder: warp prefix (in place), the chunk's count and its global base
    for (uint32_t d = threadIdx.x; d <= D; d += blockDim.x) {
      uint32_t run = 0;
#pragma unroll
      for (int w = 0; w < kWarps; ++w) {
        const uint32_t x = cnt[w * DW + d];
        cnt[w * DW + d] = run;
        run += x;
      }
      loff[d] = run;
      gbase[d] = sseg[d] + (own_offset ? off : __ldcg(offs + (size_t)d * chunks + c));
    }
    __syncthreads();
    if (!copy) {
      // only perm: each query's place is its decoder's base + its warp's
      // prefix + its rank, and the equal decoders of a 32-query group get
      // consecutive places, so the stores of a group of one decoder (most of
      // a G-buffer's) coalesce without a local sort
      if (last) pdl_trigger();  // the decode may launch (it waits for this grid before reading)
      if (one) {  // one decoder: 256 consecutive places from one base
        if (d0 <= D) {
          const uint32_t base = gbase[d0] + cnt[warp * DW + d0];
#pragma unroll
          for (int it = 0; it < kBucketItems; ++it) {
            const uint32_t p = base + it * 32 + lane;
            if (p < n) perm[p] = (uint32_t)(cbase + wbase + it * 32 + lane);
          }
        }
      } else {
#pragma unroll
        for (int it = 0; it < kBucketItems; ++it) {
          const uint32_t d = dec[it];
          const uint32_t p = d <= D ? gbase[d] + cnt[warp * DW + d] + rank[it] : 0xFFFFFFFFu;
          if (p < n) perm[p] = (uint32_t)(cbase + wbase + it * 32 + lane);
        }
      }
      __syncthreads();  // cnt and gbase are reused by the next chunk
      for (uint32_t i = threadIdx.x; i < kWarps * DW; i += blockDim.x) cnt[i] = 0;
      __syncthreads();
      continue;
    }
    block_scan(loff, D + 1);  // exclusive scan of the chunk's counts over decoders
    // stable local sort of (local index, decoder) pairs
#pragma unroll
    for (int it = 0; it < kBucketItems; ++it) {
      const uint32_t d = dec[it];
      if (d > D) continue;
      const uint32_t lp = loff[d] + cnt[warp * DW + d] + rank[it];
      sidx[lp] = (uint16_t)(wbase + it * 32 + lane);
      sdec[lp] = (uint16_t)d;
    }
    if (!FROM_Q) asm volatile("cp.async.wait_all;\n" ::: "memory");
    __syncthreads();
    if (last) pdl_trigger();  // the decode may launch (it waits for this grid before reading)
    // the counters are free again: cleared for the next chunk while this one
    // is copied out
    for (uint32_t i = threadIdx.x; i < kWarps * DW; i += blockDim.x) cnt[i] = 0;
    // coalesced copy-out of perm and the records: consecutive slots of one
    // decoder go to consecutive positions of that decoder's segment
    for (uint32_t i = threadIdx.x; i < valid; i += blockDim.x) {
      const uint32_t d = sdec[i], j = sidx[i];
      const uint32_t pos = gbase[d] + (i - loff[d]);
      if (pos < n) {
        perm[pos] = (uint32_t)(cbase + j);
        reinterpret_cast<uint4 *>(sorted)[pos] = srec[j];
      }
    }
    __syncthreads();  // srec, sidx, sdec, loff and gbase are reused by the next chunk
    if (FROM_Q && !last) {
      const size_t nb = (size_t)(c + gridDim.x) * kBucketChunk;
      stage_records(nb, (uint32_t)min((size_t)kBucketChunk, n - nb));
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

size_t bucket_chunks(size_t n) { return (n + kBucketChunk - 1) / kBucketChunk; }
size_t bucket_count_words(uint32_t D, size_t n) { return ((size_t)D + 1) * bucket_chunks(n); }
size_t bucket_meta_words(uint32_t D) { return meta_words(D) + ((size_t)D + 1) + 2; }

namespace {
template <typename DecT>
cudaError_t launch_bucket_t(const Assets &A, const ntc_query *q, size_t n, const Scratch &s, cudaStream_t st,
                            int *launches, int copy) {
  const uint32_t chunks = (uint32_t)bucket_chunks(n);
  const uint32_t D = A.num_decoders, DW = D + 2;
  const size_t smem_count = (size_t)kWarps * DW * sizeof(uint32_t);
  const size_t smem_place = (size_t)kBucketChunk * (16 + 2 + 2) + (size_t)(kWarps + 3) * DW * sizeof(uint32_t);
  const bool from_q = s.dec == nullptr;
  // k_place runs a resident grid: at most 5 CTAs per SM (its register
  // bound), fewer when its shared memory (which grows with D) allows fewer
  int dev = 0, sms = 1, smem_sm = 233472;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cudaDeviceGetAttribute(&smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev);
  size_t per_sm = (size_t)smem_sm / (smem_place + 2048);
  if (per_sm > 5) per_sm = 5;
  if (per_sm < 1) per_sm = 1;
  const uint32_t place_grid = (uint32_t)std::min<size_t>(chunks, (size_t)sms * per_sm);
  static PerDevice attrs;
  cudaError_t e = attrs.once([]() {
    // as much dynamic shared memory as the device allows a block: the
    // per-warp counters grow with the decoder count
    int dev = 0, optin = 0;
    cudaError_t r = cudaGetDevice(&dev);
    if (r == cudaSuccess) r = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    auto allow = [&](auto kernel) {
      cudaFuncAttributes fa;
      cudaError_t x = cudaFuncGetAttributes(&fa, kernel);
      if (x == cudaSuccess)
        x = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, optin - (int)fa.sharedSizeBytes);
      return x;
    };
    if (r == cudaSuccess) r = allow(k_count<DecT>);
    if (r == cudaSuccess) r = allow(k_place<DecT, false>);
    if (r == cudaSuccess) r = allow(k_place<DecT, true>);
    return r;
  });
  if (e != cudaSuccess) return e;
  *launches += 3;
  uint32_t *div_sum = s.meta + meta_words(D) + (D + 1) + 1;
  DecT *dec = reinterpret_cast<DecT *>(s.dec);
  k_count<DecT><<<chunks, kBucketThreads, smem_count, st>>>(A, q, n, chunks, s.counts, div_sum, dec);
  e = cudaGetLastError();
  if (e == cudaSuccess)
    e = launch_pdl(k_scan, dim3(D + 1), dim3(1024), 0, st, (const uint32_t *)s.counts, s.offs, chunks, D, s.meta,
                   copy);
  if (e == cudaSuccess) {
    if (from_q)
      e = launch_pdl(k_place<DecT, true>, dim3(place_grid), dim3(kBucketThreads), smem_place, st, A, q,
                     (const DecT *)nullptr, n, chunks, (const uint32_t *)s.offs, (const uint32_t *)s.meta,
                     s.perm, s.sorted);
    else
      e = launch_pdl(k_place<DecT, false>, dim3(place_grid), dim3(kBucketThreads), smem_place, st, A, q,
                     (const DecT *)dec, n, chunks, (const uint32_t *)s.offs, (const uint32_t *)s.meta, s.perm,
                     s.sorted);
  }
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}
}  // namespace

size_t bucket_dec_bytes(uint32_t D) { return D + 1 <= 256 ? 1 : 2; }

cudaError_t launch_bucket(const Assets &A, const ntc_query *q, size_t n, const Scratch &s, cudaStream_t st,
                          int *launches, int copy) {
  if (!s.dec && !copy) return cudaErrorInvalidValue;  // without the decoder array the records are always staged
  if (bucket_dec_bytes(A.num_decoders) == 1) return launch_bucket_t<uint8_t>(A, q, n, s, st, launches, copy);
  return launch_bucket_t<uint16_t>(A, q, n, s, st, launches, copy);
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
