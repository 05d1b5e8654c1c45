// tcgen05 / TMEM gather-decode (sm_103a), warp-specialised.
//
// One persistent CTA per SM runs NP producer and NC consumer warpgroups.
// Tiles (128 queries of one decoder, from the bucketing) are dealt out
// round-robin over the CTAs, so at any moment the whole GPU works on
// neighbouring tiles -- one decoder and, in set-major bucket order, one set's
// latents, which keeps them in L2.  Inside a CTA, consumer c takes the CTA's
// tiles c, c + NC, ... and is fed by its own producers through a private ring
// of SC tensor-memory stages.
//   Producer (one thread per tile row): loads the query record and its output
//     row index, computes the bilinear taps of both latent grids (Sec. 3.1, the
//     same fp32 operations as the reference addressing), fetches each bilinear
//     row as one 32-byte load from the row-pair copy of the latents, blends in
//     packed fp16 (the latents' own type) and stores the fp16/bf16 feature row
//     [16] into its stage with tcgen05.st (warp q writes TMEM lanes
//     32q..32q+31, exactly its rows).
//   Consumer: layer 1 reads A from the stage and B (the decoder's weights,
//     copied by a TMA bulk copy whenever the decoder changes) from shared
//     memory; its completion frees the stage; the ReLU/convert epilogue goes
//     TMEM -> registers -> TMEM; layers 2 and 3 read their A operand from TMEM
//     too; each layer's bias is one more K step whose A is a shared block with
//     a 1 in K column 0.  Layer 3 accumulates in the consumer's own 16 output
//     columns, so the next tile's layer 1 runs before the outputs are read;
//     the sigmoid epilogue scatters rows to out[perm[i]] (fp32, or fp16 rows).
//     At H = 64 (four consumers) one elected thread of the consumer issues its
//     MMAs.  At H = 128 (two consumers, tensor memory for no more) two issuer
//     warps per consumer issue them and hand over through named barriers, the
//     four epilogue warps only convert and write outputs, and a tile's
//     outputs are written while the next tile's layer 2 runs.
// Shared-memory B operands use the no-swizzle K-major canonical layout: 8-row
// x 16-byte core matrices, K-adjacent core matrices 128 B apart (LBO), 8-row
// groups K*16 B apart (SBO).  Every wait is bounded by time; on expiry the
// kernel records an error and stops cleanly (TMEM is always released).
//
// This header holds the kernel template; decode_tc.cu instantiates the
// production kernels and decode_tc_debug.cu the debug ones (DBG), in their own
// translation units.
#pragma once

#include "tcgen05.cuh"

namespace ntc {

constexpr int kTcKA = 32;  // K of layer 1's weight image: 16 features + the bias K step

namespace {

template <int H>
struct TcLayout {
  static constexpr uint32_t KH = H + 16;
  static constexpr uint32_t W1 = H * kTcKA * 2;
  static constexpr uint32_t W2 = H * KH * 2;
  static constexpr uint32_t W3 = 16 * KH * 2;
  static constexpr uint32_t WIMG = W1 + W2 + W3;
};

// Latent taps of one query from one mip, loaded ahead of use: 2 levels x 4
// taps; a mip blend factor is folded into the weights.
struct Taps {
  static constexpr int N = 8;
  uint4 raw[N];
  float w[N];
};

// Mip selection of one query row, kept between the two fetch phases of a
// kernel that may blend mips.
struct MipPick {
  int lo = 0;
  float t = 0.0f;
};

// One axis of the tap addressing, fp32 round-to-nearest with no contraction
// (the same operations, in the same order, as the reference addressing).
// WRAP: c is finite and the texel pair wraps at the edge; clamp: both texels
// are clamped into [0, n-1].
template <bool WRAP>
__device__ __forceinline__ void axis_pair(float c, uint32_t n, uint32_t &i0, uint32_t &i1, float &frac) {
  const float x = WRAP ? __fsub_rn(__fmul_rn(__fsub_rn(c, floorf(c)), (float)n), 0.5f)
                       : __fsub_rn(__fmul_rn(c, (float)n), 0.5f);
  const float x0f = floorf(x);
  frac = __fsub_rn(x, x0f);
  if (WRAP) {
    const int x0 = (int)x0f;  // in [-1, n-1]
    i0 = x0 < 0 ? n - 1 : (uint32_t)x0;
    const uint32_t a1 = (uint32_t)(x0 + 1);
    i1 = a1 == n ? 0u : a1;
  } else {
    const int x0 = (int)fminf(fmaxf(x0f, -1.0f), (float)n);
    i0 = (uint32_t)min(max(x0, 0), (int)n - 1);
    i1 = (uint32_t)min(x0 + 1, (int)n - 1);
  }
}

// Both texels of one bilinear row from the row-pair copy: one 32-byte load.
struct alignas(32) TexelPair {
  uint4 a, b;
};
__device__ __forceinline__ void ld_pair(const TexelPair *p, uint4 &a, uint4 &b) {
  asm volatile("ld.global.nc.v8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
               : "=r"(a.x), "=r"(a.y), "=r"(a.z), "=r"(a.w), "=r"(b.x), "=r"(b.y), "=r"(b.z), "=r"(b.w)
               : "l"(p));
}

// The texel coordinates one grid fetch used (kept only by the debug build).
struct TapIdx {
  uint32_t i0, i1, j0, j1;
};

// Issue the tap loads of one grid (taps 00, 10 from row j0; 01, 11 from row
// j1) and compute their bilinear weights, scaled by sc.  In-grid offsets are
// 32-bit (a grid holds fewer than 2^32 texels).  Clamp mode at an edge has
// x0 = x1, while the pair at x0 holds x0 and its right neighbour: the whole
// row weight then goes to the first texel.  DBG: also report the coordinates.
template <bool WRAP, bool DBG = false>
__device__ __forceinline__ void grid_fetch(const uint4 *pair, const GridDesc &g, float u, float v, float sc,
                                           uint4 *raw, float *w, TapIdx *ti = nullptr) {
  uint32_t i0, i1, j0, j1;
  float fx, fy;
  axis_pair<WRAP>(u, g.W, i0, i1, fx);
  axis_pair<WRAP>(v, g.H, j0, j1, fy);
  if (DBG) *ti = TapIdx{i0, i1, j0, j1};
  const TexelPair *p = reinterpret_cast<const TexelPair *>(pair) + g.base;
  ld_pair(p + (j0 * g.W + i0), raw[0], raw[1]);
  ld_pair(p + (j1 * g.W + i0), raw[2], raw[3]);
  const float ax = __fsub_rn(1.0f, fx), ay = __fsub_rn(1.0f, fy);
  float w00 = __fmul_rn(ax, ay), w10 = __fmul_rn(fx, ay), w01 = __fmul_rn(ax, fy), w11 = __fmul_rn(fx, fy);
  if (!WRAP && i1 == i0) {
    w00 = __fadd_rn(w00, w10);
    w01 = __fadd_rn(w01, w11);
    w10 = w11 = 0.0f;
  }
  w[0] = w00 * sc;
  w[1] = w10 * sc;
  w[2] = w01 * sc;
  w[3] = w11 * sc;
}

// All tap loads of one query from mip lo, issued before any is consumed.  A
// row that is not good (padding, bad set id or UV, bad bucket) fetches texel
// (0, 0) of set 0 instead: no branch and no out-of-range address; its flag
// marks it.  TRI: the kernel may blend mips, so the mip is selected per row
// and mip lo is weighted by 1 - t; otherwise every grid has one mip.
template <bool TRI, bool WRAP, bool DBG = false>
__device__ __forceinline__ void issue_taps(const Assets &A, const GridDesc *grids, const ntc_query &q,
                                           bool good, Taps &tp, MipPick &mp, TapIdx *ti = nullptr) {
  const uint32_t sid = good ? q.set_id : 0u;
  const float u = good ? q.u : 0.0f, v = good ? q.v : 0.0f;
  if (TRI) mp.lo = select_mip(good ? q.lod : 0.0f, A.num_mips, mp.t);
  const uint32_t M = TRI ? A.num_mips : 1u;
  const GridDesc *g = grids + (size_t)sid * kLevels * M;
  const float s = TRI ? __fsub_rn(1.0f, mp.t) : 1.0f;
#pragma unroll
  for (int k = 0; k < kLevels; ++k)
    grid_fetch<WRAP, DBG>(A.pair, g[k * M + mp.lo], u, v, s, tp.raw + 4 * k, tp.w + 4 * k, DBG ? ti + k : nullptr);
}

// The second phase of a mip blend, one level at a time (fewer registers live
// than a whole query's taps): the taps of level k at mip lo + 1, weighted by
// t, for the rows with t > 0 (the others load nothing and get zero weights, so
// their accumulation is unchanged).
template <bool WRAP, bool DBG = false>
__device__ __forceinline__ void issue_level_hi(const Assets &A, const GridDesc *grids, const ntc_query &q,
                                               bool good, const MipPick &mp, int k, uint4 (&raw)[4],
                                               float (&w)[4], TapIdx *ti = nullptr) {
  if (good && mp.t > 0.0f) {
    const uint32_t M = A.num_mips;
    grid_fetch<WRAP, DBG>(A.pair, grids[((size_t)q.set_id * kLevels + k) * M + mp.lo + 1], q.u, q.v, mp.t, raw, w,
                          ti);
  } else {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      w[i] = 0.0f;
      raw[i] = make_uint4(0, 0, 0, 0);
    }
  }
}

// acc[c/2] += w * tap[c] over the 8 channels of one tap, in packed fp16 pairs
// (the latents' own type; hfma2, the first tap multiplies): the feature row
// becomes the fp16/bf16 A operand, so the blend needs no fp32 conversions.
template <bool FIRST>
__device__ __forceinline__ void accum_tap_x2(__half2 (&acc)[4], uint4 raw, float w) {
  const __half2 ww = __float2half2_rn(w);
  const __half2 *h = reinterpret_cast<const __half2 *>(&raw);
#pragma unroll
  for (int p = 0; p < 4; ++p) acc[p] = FIRST ? __hmul2(ww, h[p]) : __hfma2(ww, h[p], acc[p]);
}

// Feature accumulation: acc[k][c/2] over the 8 channels of level k, all taps
// of mip lo first (FIRST: the first tap multiplies), then those of mip lo + 1.
template <bool FIRST>
__device__ __forceinline__ void accum_taps(const Taps &tp, __half2 (&acc)[kLevels][4]) {
#pragma unroll
  for (int k = 0; k < kLevels; ++k) {
    accum_tap_x2<FIRST>(acc[k], tp.raw[k * 4], tp.w[k * 4]);
#pragma unroll
    for (int p = 1; p < 4; ++p) accum_tap_x2<false>(acc[k], tp.raw[k * 4 + p], tp.w[k * 4 + p]);
  }
}

template <bool BF16>
__device__ __forceinline__ void pack_row(const __half2 (&acc)[kLevels][4], uint32_t (&packed)[8]) {
#pragma unroll
  for (int k = 0; k < kLevels; ++k)
#pragma unroll
    for (int p = 0; p < 4; ++p) {
      if (BF16) {
        const float2 x = __half22float2(acc[k][p]);
        packed[k * 4 + p] = pack<true>(x.x, x.y);
      } else {
        packed[k * 4 + p] = *reinterpret_cast<const uint32_t *>(&acc[k][p]);
      }
    }
}

__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void *src, uint32_t bytes, uint32_t bar) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(bar), "r"(bytes) : "memory");
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];\n" ::"r"(dst),
      "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}

constexpr uint32_t kSmemTileTable = 1024;  // staged when D + 2 <= this
constexpr uint32_t kSmemGrids = 1024;      // staged when S * 2 * M <= this


// Shared-memory plan of the warp-specialised kernel: only the decoders' weights
// (the B operands) and bookkeeping live in shared memory; every A operand and
// accumulator lives in tensor memory, so most of the SM's L1/shared array stays
// L1, which holds the in-flight latent gathers.
// Whether each consumer has MMA-issuing warps of its own.  One thread issues
// a tcgen05.mma about every 65-90 cycles whatever N is (two warps issue in
// parallel; two lanes of one warp barely do), so at H = 128 (20 MMAs a tile)
// a consumer warpgroup that issued its own MMAs would spend about a third of
// each tile issuing while its other warps wait.  With issuer warps the four
// epilogue warps only convert accumulators and write outputs.  Issuer A
// issues layers 1 and 2 and prepares the next tile while layer 2's result is
// converted; issuer B issues the output layer, its first K steps while the
// second half of its operand is still being converted, its last ones while A
// issues the next tile's layer 1.  The H = 64 kernel (four consumers, 1024
// threads) has no registers to spare for the extra warps.
template <int H>
__host__ __device__ constexpr bool issuer_warp() {
  return H >= 128;
}

// Named barriers between a consumer's epilogue warps (E) and its issuers A and
// B (ids above the warpgroup barriers 1..NP+NC), with their thread counts:
// T A hands a tile over to E and B (192), X E has converted layer 1's result,
// or taken over a tile with nothing to multiply (A waits, 160), Y E has
// converted the first half of layer 2's result and read the previous tile's
// outputs (B waits, 160), Z E has converted all of it (A and B wait, 192).  X,
// Y and Z of a tile with nothing to multiply: only X.
constexpr int kIssT = 0, kIssX = 1, kIssY = 2, kIssZ = 3;
constexpr int kIssTN = 192, kIssXN = 160, kIssYN = 160, kIssZN = 192;
template <int NP, int NC>
__device__ __forceinline__ int iss_bar(int c, int which) {
  return NP + NC + 1 + 4 * c + which;
}
__device__ __forceinline__ void named_sync(int id, int n) {
  asm volatile("bar.sync %0, %1;\n" ::"r"(id), "r"(n) : "memory");
}
__device__ __forceinline__ void named_arrive(int id, int n) {
  asm volatile("bar.arrive %0, %1;\n" ::"r"(id), "r"(n) : "memory");
}

template <int H, int NC, int SC>
struct TmSmem {
  using L = TcLayout<H>;
  static constexpr int S = NC * SC;                                     // stages in all rings
  static constexpr size_t weights = 0;                                  // per consumer
  // per stage and use parity: 128 output rows, 0xFFFFFFFF for a row that is
  // not good (never a valid row: n <= 2^32 - 256).  Two slots per stage: the
  // producer's next use of a stage writes the other slot, so a consumer warp
  // that reads late never sees the following tile's rows.
  static constexpr size_t oidx = weights + (size_t)NC * L::WIMG;
  static constexpr size_t bars = oidx + (size_t)S * 2 * 128 * 4;
  // full, empty, mma, weights, output; with issuer warps each issuer's final commit
  static constexpr int nbars = 2 * S + 3 * NC + (issuer_warp<H>() ? 2 * NC : 0);
  static constexpr size_t misc = bars + (size_t)nbars * 8;
  static constexpr size_t tiles = misc + 64;
  static constexpr size_t grids = tiles + 2 * kSmemTileTable * 4;
  static constexpr size_t total = grids + kSmemGrids * sizeof(GridDesc);
};

// Tensor-memory plan (columns).  The NC fp32 accumulators (H columns each)
// come first, so every accumulator starts on a multiple of H; then each
// consumer's hidden A operand (H/2 columns: two 16-bit K elements per column);
// then the layer-1 feature operands [128 x 16] of the NC * SC ring stages (8
// columns each); last, one shared 8-column block holding a 1 in K column 0 and
// zeros elsewhere: the A operand of every layer's bias K step (the decoder image
// keeps each layer's bias as the first row of an extra 16-row K block); then
// each consumer's own 16-column accumulator for the output layer, so that the
// next tile's layer 1 can run in the hidden accumulator meanwhile.

template <int H, int NC, int SC>
struct TmCols {
  static constexpr uint32_t HID = NC * H;
  static constexpr uint32_t STG = HID + NC * (H / 2);
  static constexpr uint32_t ONES = STG + NC * SC * 8;
  static constexpr uint32_t OUT = (ONES + 8 + 15) / 16 * 16;
  static constexpr uint32_t used = OUT + NC * 16;
  static constexpr uint32_t alloc = used <= 256 ? 256 : 512;
  static_assert(used <= 512, "tensor memory plan exceeds 512 columns");
  static __device__ __forceinline__ uint32_t acc(uint32_t c) { return c * H; }
  static __device__ __forceinline__ uint32_t hid(uint32_t c) { return HID + c * (H / 2); }
  // layer-1 A operand of stage s (= consumer * SC + st)
  static __device__ __forceinline__ uint32_t a1(uint32_t s) { return STG + 8 * s; }
  static __device__ __forceinline__ uint32_t out(uint32_t c) { return OUT + 16 * c; }
};

// Warp-specialised gather-decode with tensor-memory operands.
//   Consumer warpgroups (the last NC) each decode the CTA's local tiles
//   k = c, c + NC, ... (j = k / NC counts a consumer's tiles).  Each consumer has
//   a private ring of SC stages in tensor memory, filled by its own R = NP / NC
//   producer warpgroups: tile j of consumer c is gathered by producer c + NC *
//   (j mod R) into stage j mod SC.  SC is a multiple of R, so every stage has one
//   producer and one consumer and successive uses of a stage are ordered by
//   program order on both sides -- an mbarrier parity wait can then never be two
//   phases ahead of its barrier.
//   Producer: each thread computes the taps of one query row, blends them in
//   packed fp16 and stores the fp16/bf16 feature row into the stage's TMEM A
//   region (tcgen05.st; warp q of a warpgroup owns TMEM lanes 32q..32q+31,
//   exactly its rows), with the row's output index (or 0xFFFFFFFF if the row is
//   not good) in shared memory, in the slot of the stage's use parity; four
//   warp arrivals fill the stage.  The next tile's query record and output
//   index are loaded while the current tile is gathered.
//   Consumer: layer 1 reads A from the stage and B (weights) from shared memory;
//   its completion empties the stage; the ReLU/convert epilogue goes TMEM ->
//   registers -> TMEM; layers 2 and 3 read their A from TMEM too.  Layer 3
//   writes the consumer's own output columns and completes on its own
//   barrier, so the next tile's layer 1 is issued first; then the sigmoid
//   epilogue scatters rows to out[perm[i]].
// CTA b owns the global tiles b, b + grid, b + 2 grid, ...
// DBG (a separate instantiation, for tests): every producer also records the
// row it built -- texel indices, the 16 bytes blended for each tap, their
// weights, the mip pick and the packed feature row -- in dbg[output row].
template <int H, bool BF16, bool TRI, bool WRAP, int CP, int NP, int NC, int SC, bool DBG>
__global__ void __launch_bounds__((NP + NC) * 128 + (issuer_warp<H>() ? NC * 64 : 0), 1)
    k_decode_tm(Assets A, WeightImages W, Buckets B, void *out, unsigned long long *err,
                unsigned int *status, int vec_out, ntc_debug_row *dbg) {
  static_assert(NP % NC == 0 && SC % (NP / NC) == 0, "each ring stage needs one producer");
  constexpr int R = NP / NC;  // producers per consumer
  constexpr bool ISS = issuer_warp<H>();
  constexpr int S = NC * SC;
  using L = TcLayout<H>;
  using M = TmSmem<H, NC, SC>;
  using TC = TmCols<H, NC, SC>;
  extern __shared__ __align__(128) uint8_t smem[];
  const int role = threadIdx.x >> 7, row = threadIdx.x & 127, warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t lanes = (uint32_t)((warp & 3) * 32) << 16;  // this warp's TMEM lane quadrant
  const uint32_t sbase = saddr(smem);
  uint64_t *bars = reinterpret_cast<uint64_t *>(smem + M::bars);
  auto full_bar = [&](uint32_t s) { return saddr(bars + s); };
  auto empty_bar = [&](uint32_t s) { return saddr(bars + S + s); };
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + M::misc);
  volatile uint32_t *abort_flag = tmem_slot + 1;
  // [NC][2]: consumer c's decision to stop, written for its tile jc in slot jc & 1
  volatile uint32_t *stop_flag = tmem_slot + 2;
  const uint32_t D = A.num_decoders, C = W.out_dim;

  // no stage has rows yet: a consumer that stops on a wait timeout reads
  // all-bad rows, never an uninitialised output index
  for (uint32_t i = threadIdx.x; i < (uint32_t)S * 2 * 128; i += blockDim.x)
    reinterpret_cast<uint32_t *>(smem + M::oidx)[i] = 0xFFFFFFFFu;
  const GridDesc *grids = A.pgrids;  // grid bases in the row-pair copy
  const uint32_t ngrids = A.num_sets * kLevels * A.num_mips;
  if (ngrids <= kSmemGrids) {
    GridDesc *s_grids = reinterpret_cast<GridDesc *>(smem + M::grids);
    for (uint32_t i = threadIdx.x; i < ngrids; i += blockDim.x) s_grids[i] = A.pgrids[i];
    grids = s_grids;
  }
  if (threadIdx.x == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(full_bar(i), 4);   // one arrival per producer warp
      mbar_init(empty_bar(i), 1);  // the consumer's layer-1 commit
    }
    for (int i = 2 * S; i < M::nbars; ++i) mbar_init(saddr(bars + i), 1);
    *abort_flag = 0;
    for (int i = 0; i < 2 * NC; ++i) stop_flag[i] = 0;
    asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(
                     saddr(tmem_slot)),
                 "r"(TC::alloc)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
  }
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const uint32_t one = BF16 ? 0x3F80u : 0x3C00u;  // 1.0 in the low half, 0 in the high half
  if (warp < 4) {  // the shared bias operand: K column 0 is 1, the rest 0
    const uint32_t z[8] = {one, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
    tmem_st8(tmem_base + TC::ONES + lanes, z);
    tmem_wait_st();
  }
  // everything above is independent of the bucketing; the tile table is not
  pdl_wait();
  const uint32_t *seg = B.meta + 1, *tst = B.meta + 1 + (D + 2);
  if (!B.identity_n && D + 2 <= kSmemTileTable) {
    uint32_t *s_seg = reinterpret_cast<uint32_t *>(smem + M::tiles);
    uint32_t *s_tst = s_seg + kSmemTileTable;
    for (uint32_t i = threadIdx.x; i < D + 2; i += blockDim.x) {
      s_seg[i] = __ldg(seg + i);
      s_tst[i] = __ldg(tst + i);
    }
    seg = s_seg;
    tst = s_tst;
  }
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t T = B.identity_n ? (B.identity_n + kTile - 1) / kTile : __ldg(B.meta);
  const uint32_t grid = gridDim.x;
  const uint32_t K = blockIdx.x < T ? (T - blockIdx.x + grid - 1) / grid : 0;  // local tiles

  if (role < NP) {
    // ------------------------------------------------------------ producer
    const uint32_t pc = role % NC, pq = role / NC;  // serves consumer pc, tiles j = pq mod R
    auto tile_of = [&](uint32_t j) { return pc + NC * j; };
    uint32_t j = pq;
    // Records read through perm (the caller's array, when the bucketing did
    // not copy them): the output rows are loaded two tiles ahead and the
    // query records one tile ahead, so a record never waits on its own perm
    // load (DEEP; the H = 64 kernels that blend mips have no registers to
    // spare for it).  Otherwise a row's output row and record are loaded
    // together, one tile ahead.
    constexpr bool DEEP = H > 64 || !TRI;
    const bool copied = rows_copied(B, D);
    const bool two_stage = DEEP && !copied;
    TileWalk walk;
    walk.ident_n = B.identity_n;
    // this thread's row of the producer's tile jj: its output row, or kNoRow
    // past the tile's end.  A row of the bad bucket (set id out of range)
    // needs no flag of its own: query_bad() rejects it.
    constexpr uint32_t kNoRow = 0xFFFFFFFFu;  // never a row: n <= 2^32 - 256
    auto out_row = [&](uint32_t jj) -> uint32_t {
      if (tile_of(jj) >= K) return kNoRow;
      uint32_t d_, st_, len_;
      walk.at(seg, tst, D, blockIdx.x + tile_of(jj) * grid, d_, st_, len_);
      if ((uint32_t)row >= len_) return kNoRow;
      return B.identity_n ? st_ + row : __ldg(B.perm + st_ + row);
    };
    // one stage: the row's output row and query record together
    auto fetch_row = [&](uint32_t jj, uint32_t &oi_, ntc_query &q_) {
      oi_ = kNoRow;
      if (tile_of(jj) >= K) return;
      uint32_t d_, st_, len_;
      walk.at(seg, tst, D, blockIdx.x + tile_of(jj) * grid, d_, st_, len_);
      if ((uint32_t)row < len_) bucket_row(B, copied, st_ + row, oi_, q_);
    };
    uint32_t oi, noi = kNoRow;
    ntc_query q;
    if (two_stage) {
      oi = out_row(j);
      noi = out_row(j + R);
      if (oi != kNoRow) q = load_query(B.queries + oi);
    } else {
      fetch_row(j, oi, q);
    }
    for (; tile_of(j) < K; j += R) {
      if (*abort_flag) break;
      // the next tile's query record (and, two-stage, the output row of the
      // tile after it) go in flight early: before the taps, or (TRI, where
      // registers are scarcer) once the first mip's taps are consumed
      uint32_t nnoi = kNoRow;
      ntc_query nq;
      auto prefetch = [&]() {
        if (two_stage) {
          if (noi != kNoRow) nq = load_query(B.queries + noi);
          nnoi = out_row(j + 2 * R);
        } else {
          fetch_row(j + R, noi, nq);
        }
      };
      if (!TRI) prefetch();
      const bool valid = oi != kNoRow;
      const bool good = valid && !query_bad(A, q);
      Taps taps;
      MipPick mp;
      TapIdx ti[kLevels];
      issue_taps<TRI, WRAP, DBG>(A, grids, q, good, taps, mp, ti);
      // the record of a debug build: texel (i, j) of grid (set, level, mip) is
      // texel base + j * W + i of the caller's latents
      auto record = [&](int k, int slot, const uint4 *raw, const float *w, const TapIdx &x) {
        ntc_debug_row &r = dbg[oi];
        const GridDesc gl = A.grids[((size_t)q.set_id * kLevels + k) * A.num_mips + mp.lo + slot];
        const unsigned long long r0 = gl.base + (unsigned long long)x.j0 * gl.W;
        const unsigned long long r1 = gl.base + (unsigned long long)x.j1 * gl.W;
        r.idx[k][slot][0] = r0 + x.i0;
        r.idx[k][slot][1] = r0 + x.i1;
        r.idx[k][slot][2] = r1 + x.i0;
        r.idx[k][slot][3] = r1 + x.i1;
#pragma unroll
        for (int p = 0; p < 4; ++p) {
          r.raw[k][slot][p][0] = raw[p].x;
          r.raw[k][slot][p][1] = raw[p].y;
          r.raw[k][slot][p][2] = raw[p].z;
          r.raw[k][slot][p][3] = raw[p].w;
          r.w[k][slot][p] = w[p];
        }
      };
      if (DBG && good) {
        dbg[oi].t = mp.t;
        dbg[oi].lo = (uint32_t)mp.lo;
#pragma unroll
        for (int k = 0; k < kLevels; ++k) record(k, 0, taps.raw + 4 * k, taps.w + 4 * k, ti[k]);
      }
      // bad rows (set id out of range, non-finite UV, or the bad bucket) decode to NaN
      const bool bad = valid && !good;
      const uint32_t badm = __ballot_sync(0xFFFFFFFFu, bad);
      if (badm && lane == __ffs(badm) - 1) atomicAdd(err, (unsigned long long)__popc(badm));
      if (bad) put_nan_row(out, oi, C, W.out_half);
      __half2 acc[kLevels][4];
      accum_taps<true>(taps, acc);
      if (TRI) prefetch();
      if (TRI && __any_sync(0xFFFFFFFFu, good && mp.t > 0.0f)) {  // some row blends two mips
#pragma unroll
        for (int k = 0; k < kLevels; ++k) {
          uint4 raw[4];
          float w[4];
          TapIdx th;
          issue_level_hi<WRAP, DBG>(A, grids, q, good, mp, k, raw, w, &th);
          if (DBG && good && mp.t > 0.0f) record(k, 1, raw, w, th);
#pragma unroll
          for (int p = 0; p < 4; ++p) accum_tap_x2<false>(acc[k], raw[p], w[p]);
        }
      }
      uint32_t a[8];
      pack_row<BF16>(acc, a);
      if (DBG && good)
#pragma unroll
        for (int i = 0; i < 8; ++i) dbg[oi].feat[i] = a[i];
      const uint32_t s = pc * SC + j % SC, n = j / SC;
      if (!mbar_wait(empty_bar(s), (n & 1) ^ 1)) {  // the stage's previous tile has left layer 1
        atomicOr(status, 1u);
        *abort_flag = 1;
      }
      fence_after();
      tmem_st8(tmem_base + TC::a1(s) + lanes, a);
      tmem_wait_st();
      reinterpret_cast<uint32_t *>(smem + M::oidx)[(s * 2 + (n & 1)) * 128 + row] = good ? oi : 0xFFFFFFFFu;
      fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(full_bar(s));
      q = nq;
      oi = noi;
      if (two_stage) noi = nnoi;
    }
  } else if (role < NP + NC) {
    // ------------------------------------------------------------ consumer
    const int c = role - NP;
    const int wgid = role;  // named barrier id role + 1
    const bool poller = (row >> 5) == (c & 3);  // one waiting warp per consumer, spread over the sub-partitions
    const uint32_t tD = tmem_base + TC::acc(c);  // accumulator
    const uint32_t tH = tmem_base + TC::hid(c);  // hidden A operand
    const uint32_t tOnes = tmem_base + TC::ONES; // the bias K step's A operand
    const uint32_t tO = tmem_base + TC::out(c);  // the output layer's accumulator
    const uint32_t sW1 = sbase + (uint32_t)(M::weights + c * L::WIMG), sW2 = sW1 + L::W1, sW3 = sW2 + L::W2;
    const uint32_t mbar = saddr(bars + 2 * S + c), wbar = saddr(bars + 2 * S + NC + c);
    const uint32_t obar = saddr(bars + 2 * S + 2 * NC + c);  // the output layer's completion
    uint32_t ph = 0, wph = 0, oph = 0, cur = 0xFFFFFFFFu;
    TileWalk cwalk;
    cwalk.ident_n = B.identity_n;
    constexpr uint32_t id_hidden = instr_desc<BF16>(H), id_out = instr_desc<BF16>(16);
    const uint64_t dW1 = smem_desc(sW1, kTcKA), dW2 = smem_desc(sW2, L::KH), dW3 = smem_desc(sW3, L::KH);
    auto wait_bar = [&](uint32_t b, uint32_t parity) {
      if (poller && !mbar_wait(b, parity)) {
        atomicOr(status, 1u);
        *abort_flag = 1;
      }
    };
    // TMEM accumulator columns [c_lo, c_hi) -> ReLU -> fp16/bf16 pairs -> hidden A operand
    auto hidden = [&](int c_lo = 0, int c_hi = H) {
#pragma unroll 1
      for (int c0 = c_lo; c0 < c_hi; c0 += 32) {
        uint32_t v[32];
        tmem_ld32(tD + lanes + c0, v);
        tmem_wait_ld();
        uint32_t p[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) p[i] = pack_relu<BF16>(v[2 * i], v[2 * i + 1]);
        tmem_st16(tH + lanes + c0 / 2, p);
      }
      tmem_wait_st();
    };
    // Start tile k: its decoder's weights, wait for its A stage (with the
    // rows' output indices) and issue layer 1.  Requires this consumer's
    // previous tile to have read its hidden accumulator.  Its output layer may
    // still run: it reads the hidden operand and W3 of the weight image and
    // writes only tO.  So when tile k needs another decoder, that output layer
    // is waited for before the copy overwrites the image (out_pending: an
    // output layer was issued and not yet waited for).  The barrier also
    // carries the decision to stop, the same for every warp.
    bool out_pending = false;
    auto begin = [&](uint32_t k, uint32_t &dec, uint32_t &oi, bool &good, bool &stop) {
      const uint32_t jc = k / NC, t = blockIdx.x + k * grid, s = c * SC + jc % SC, n = jc / SC;
      uint32_t start, len;
      cwalk.at(seg, tst, D, t, dec, start, len);
      bool wpend = false;
      if (dec < D && dec != cur) {
        if (out_pending) {  // W3 may still be read by the previous tile's output layer
          wait_bar(obar, oph);
          oph ^= 1;
          out_pending = false;
          wg_bar(wgid);
        }
        if (row == 0) {
          fence_after();
          bulk_g2s(sW1, W.tc + (size_t)dec * W.tc_stride, L::WIMG, wbar);
        }
        wpend = true;
        cur = dec;
      }
      wait_bar(full_bar(s), n & 1);
      if (wpend) {
        wait_bar(wbar, wph);
        wph ^= 1;
      }
      if (row == 0) stop_flag[2 * c + (jc & 1)] = *abort_flag;
      wg_bar(wgid);
      stop = stop_flag[2 * c + (jc & 1)] != 0;
      oi = reinterpret_cast<const uint32_t *>(smem + M::oidx)[(s * 2 + (n & 1)) * 128 + row];
      good = oi != 0xFFFFFFFFu;
      if (row == 0) {
        fence_after();
        if (dec < D) {
          const uint32_t tA = tmem_base + TC::a1(s);
          umma_ta(tD, tA, dW1, id_hidden, 0);
          umma_ta(tD, tOnes, dW1 + 16, id_hidden, 1);  // + bias
          umma_commit(mbar);
          umma_commit(empty_bar(s));
        } else {
          mbar_arrive(empty_bar(s));  // a tile of bad queries: nothing to multiply
        }
      }
    };
    // the sigmoid epilogue of one tile: its output accumulator(s) -> out[eoi]
    auto out_rows = [&](uint32_t eoi, bool egood) {
      uint32_t o[16];
      tmem_ld16(tO + lanes, o);
      tmem_wait_ld();
      fence_before();
      if (egood) {
        // sigmoid(x) = 0.5 + 0.5 * tanh(x / 2)
        float y[CP];
#pragma unroll
        for (int cc = 0; cc < CP; ++cc) {
          float th;
          asm("tanh.approx.f32 %0, %1;" : "=f"(th) : "f"(0.5f * __uint_as_float(o[cc])));
          y[cc] = fmaf(0.5f, th, 0.5f);
        }
        if (CP == 8 && vec_out && C == 8 && W.out_half) {  // one 16-byte store per row
          uint32_t h[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const __half2 p = __floats2half2_rn(y[2 * i], y[2 * i + 1]);
            h[i] = *reinterpret_cast<const uint32_t *>(&p);
          }
          asm volatile("st.global.v4.b32 [%0], {%1, %2, %3, %4};\n" ::"l"(reinterpret_cast<__half *>(out) +
                                                                        (size_t)eoi * 8),
                       "r"(h[0]), "r"(h[1]), "r"(h[2]), "r"(h[3])
                       : "memory");
        } else if (CP == 8 && vec_out && C == 8) {  // one 32-byte store per row
          asm volatile("st.global.v8.f32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};\n" ::"l"(
                           reinterpret_cast<float *>(out) + (size_t)eoi * 8),
                       "f"(y[0]), "f"(y[1]), "f"(y[2]), "f"(y[3]), "f"(y[4]), "f"(y[5]), "f"(y[6]), "f"(y[7])
                       : "memory");
        } else {
#pragma unroll
          for (int cc = 0; cc < CP; ++cc)
            if (cc < (int)C) put_out(out, (size_t)eoi * C + cc, y[cc], W.out_half);
        }
      }
    };
    if constexpr (ISS) {
      // The epilogue warps of a consumer with issuer warps.  Per tile: A's
      // arrival on T hands the tile over (its rows' output indices, the
      // decision to stop); layer 1's result is converted (arrive on X); the
      // previous tile's outputs are written while layer 2 runs; layer 2's
      // result is converted in two halves (arrive on Y, then on Z), and B
      // issues the output layer's first K steps in between.  A tile's outputs
      // wait in tO until the next tile's layer 2.  Layer 1's result is
      // converted only once the previous output layer, which reads the hidden
      // operand, has completed.
      const int bT = iss_bar<NP, NC>(c, kIssT), bX = iss_bar<NP, NC>(c, kIssX);
      const int bY = iss_bar<NP, NC>(c, kIssY), bZ = iss_bar<NP, NC>(c, kIssZ);
      bool epi = false;    // a tile's outputs wait in tO
      bool opend = false;  // an output layer was issued and not yet waited for
      bool stopped = false;
      uint32_t poi = 0;
      bool pgood = false;
      for (uint32_t k = c; k < K; k += NC) {
        const uint32_t jc = k / NC, t = blockIdx.x + k * grid, s = c * SC + jc % SC, n = jc / SC;
        uint32_t dec, start, len;
        cwalk.at(seg, tst, D, t, dec, start, len);
        named_sync(bT, kIssTN);
        if (stop_flag[2 * c + (jc & 1)]) {
          stopped = true;
          break;
        }
        const uint32_t oi = reinterpret_cast<const uint32_t *>(smem + M::oidx)[(s * 2 + (n & 1)) * 128 + row];
        const bool good = oi != 0xFFFFFFFFu;
        if (dec < D) {
          wait_bar(mbar, ph);  // layer 1
          ph ^= 1;
          if (opend) {  // the previous output layer has read the hidden operand
            wait_bar(obar, oph);
            oph ^= 1;
            opend = false;
          }
          wg_bar(wgid);
          fence_after();
          hidden();
          fence_before();
          named_arrive(bX, kIssXN);
          if (epi) {
            out_rows(poi, pgood);
            epi = false;
          }
          wait_bar(mbar, ph);  // layer 2
          ph ^= 1;
          wg_bar(wgid);
          fence_after();
          hidden(0, H / 2);
          fence_before();
          named_arrive(bY, kIssYN);
          hidden(H / 2, H);
          fence_before();
          named_arrive(bZ, kIssZN);
          epi = true;
          opend = true;
          poi = oi;
          pgood = good;
        } else {  // a tile with nothing to multiply
          named_arrive(bX, kIssXN);  // taken over: A may hand over the next tile
          if (epi) {                 // write the waiting outputs now
            if (opend) {
              wait_bar(obar, oph);
              oph ^= 1;
              opend = false;
            }
            wg_bar(wgid);
            fence_after();
            out_rows(poi, pgood);
            epi = false;
          }
        }
      }
      if (epi && !stopped) {  // the last tile's outputs
        if (opend) wait_bar(obar, oph);
        wg_bar(wgid);
        fence_after();
        out_rows(poi, pgood);
      }
    } else {
      uint32_t k = c, dec = D, oi = 0;
      bool good = false, stop = false;
      if (k < K) begin(k, dec, oi, good, stop);
      while (k < K) {
        if (dec < D) {
#pragma unroll 1
          for (int layer = 0; layer < 2; ++layer) {
            wait_bar(mbar, ph);
            ph ^= 1;
            wg_bar(wgid);
            fence_after();
            hidden();
            fence_before();
            wg_bar(wgid);
            if (row == 0) {
              fence_after();
              if (layer == 0) {
#pragma unroll
                for (uint32_t kq = 0; kq < H / 16; ++kq) umma_ta(tD, tH + 8 * kq, dW2 + 16 * kq, id_hidden, kq);
                umma_ta(tD, tOnes, dW2 + 16 * (H / 16), id_hidden, 1);  // + bias
                umma_commit(mbar);
              } else {
#pragma unroll
                for (uint32_t kq = 0; kq < H / 16; ++kq) umma_ta(tO, tH + 8 * kq, dW3 + 16 * kq, id_out, kq);
                umma_ta(tO, tOnes, dW3 + 16 * (H / 16), id_out, 1);  // + bias
                umma_commit(obar);
              }
            }
          }
          out_pending = true;
        }
        // the next tile's layer 1 runs while this tile's output layer finishes
        // and its outputs are written (the hidden accumulator has been read)
        const uint32_t kn = k + NC;
        uint32_t ndec = D, noi = 0;
        bool ngood = false, nstop = false;
        if (kn < K && !stop) begin(kn, ndec, noi, ngood, nstop);
        if (dec < D) {
          if (out_pending) {  // not already waited for by begin()
            wait_bar(obar, oph);
            oph ^= 1;
            out_pending = false;
          }
          wg_bar(wgid);
          fence_after();
          out_rows(oi, good);
        }
        if (stop || nstop) {  // every warp of this warpgroup read the same flags
          if (nstop && ndec < D) wait_bar(mbar, ph);  // the issued layer 1 ends before TMEM is released
          break;
        }
        k = kn;
        dec = ndec;
        oi = noi;
        good = ngood;
      }
    }
  } else if constexpr (ISS) {
    // ------------------------------------------------------------ MMA issuers
    // Warps 2c (A) and 2c + 1 (B) after the warpgroups issue consumer c's
    // MMAs (lane 0).  A prepares each tile -- waits for the stage's features
    // and, when the decoder changes, for the previous output layer (it reads
    // W3 of the image the copy replaces) and the new weights -- and hands it
    // over on T with the decision to stop, so every warp of the consumer
    // stops at the same tile.  A issues layer 1, layer 2 once X arrives, and
    // prepares the next tile while the epilogue converts layer 2's result; B
    // issues the output layer's bias and first K steps once Y arrives and the
    // rest once Z arrives.  Every wait is bounded.
    const int iw = (int)((threadIdx.x - (NP + NC) * 128) >> 5);
    const int c = iw >> 1;
    const bool issuer_a = (iw & 1) == 0;
    const uint32_t tD = tmem_base + TC::acc(c), tH = tmem_base + TC::hid(c), tOnes = tmem_base + TC::ONES;
    const uint32_t tO = tmem_base + TC::out(c);
    const uint32_t sW1 = sbase + (uint32_t)(M::weights + c * L::WIMG), sW2 = sW1 + L::W1, sW3 = sW2 + L::W2;
    const uint32_t mbar = saddr(bars + 2 * S + c), wbar = saddr(bars + 2 * S + NC + c);
    const uint32_t obar = saddr(bars + 2 * S + 2 * NC + c);
    const uint32_t fbar = saddr(bars + 2 * S + 3 * NC + 2 * c + (issuer_a ? 0 : 1));
    const int bT = iss_bar<NP, NC>(c, kIssT), bX = iss_bar<NP, NC>(c, kIssX);
    const int bY = iss_bar<NP, NC>(c, kIssY), bZ = iss_bar<NP, NC>(c, kIssZ);
    constexpr uint32_t id_hidden = instr_desc<BF16>(H), id_out = instr_desc<BF16>(16);
    const uint64_t dW1 = smem_desc(sW1, kTcKA), dW2 = smem_desc(sW2, L::KH), dW3 = smem_desc(sW3, L::KH);
    bool issued = false;
    auto wait = [&](uint32_t b, uint32_t parity) {  // lane 0
      if (!mbar_wait(b, parity)) {
        atomicOr(status, 1u);
        *abort_flag = 1;
      }
    };
    TileWalk iwalk;
    iwalk.ident_n = B.identity_n;
    if (issuer_a) {
      uint32_t cur = 0xFFFFFFFFu, wph = 0, l3 = 0;  // l3: output layers issued (by B)
      // Tile k's stage holds its features; returns the decision to stop
      // (lane 0's, not yet shared) and whether the weights must be replaced
      // first, which waits for the previous output layer and so is left for
      // after Z.
      auto prepare = [&](uint32_t k, uint32_t &dec, bool &swap) -> uint32_t {
        const uint32_t jc = k / NC, t = blockIdx.x + k * grid, s = c * SC + jc % SC, n = jc / SC;
        uint32_t start, len;
        iwalk.at(seg, tst, D, t, dec, start, len);
        swap = dec < D && dec != cur;
        uint32_t stop = 0;
        if (lane == 0) {
          wait(full_bar(s), n & 1);  // the features and the rows' output indices
          stop = *abort_flag;
        }
        return stop;
      };
      auto load_weights = [&](uint32_t dec) {  // lane 0
        if (l3) wait(obar, (l3 - 1) & 1);
        fence_after();
        bulk_g2s(sW1, W.tc + (size_t)dec * W.tc_stride, L::WIMG, wbar);
        wait(wbar, wph);
        wph ^= 1;
      };
      uint32_t dec = D;
      bool swap = false;
      // Hands tile k over on T: the decision to stop (after the weights, if
      // the decoder changes) in the slot of the tile's parity.  An arrival on
      // T always follows this issuer's wait on X of the previous tile, which
      // the epilogue warps pass only after T of that tile has completed, so
      // two arrivals of this warp never meet in one barrier phase.  (Handing
      // the next tile over before Z was slower: the epilogue warps then poll
      // layer 1's barrier instead of waiting on T.)
      auto hand_over = [&](uint32_t k, uint32_t stop) -> uint32_t {
        const uint32_t jc = k / NC;
        if (lane == 0) {
          if (swap && !stop && !*abort_flag) load_weights(dec);
          stop |= *abort_flag;
          stop_flag[2 * c + (jc & 1)] = stop;
        }
        if (swap) cur = dec;
        stop = __shfl_sync(0xFFFFFFFFu, stop, 0);
        named_arrive(bT, kIssTN);
        return stop;
      };
      uint32_t stop = c < K ? prepare(c, dec, swap) : 0;
      for (uint32_t k = c; k < K; k += NC) {
        const uint32_t jc = k / NC, s = c * SC + jc % SC;
        stop = hand_over(k, stop);
        if (stop) break;
        const uint32_t tdec = dec;
        if (tdec < D) {
          if (lane == 0) {
            fence_after();
            umma_ta(tD, tmem_base + TC::a1(s), dW1, id_hidden, 0);
            umma_ta(tD, tOnes, dW1 + 16, id_hidden, 1);  // + bias
            umma_commit(mbar);
            umma_commit(empty_bar(s));
          }
          issued = true;
        } else if (lane == 0) {
          mbar_arrive(empty_bar(s));  // a tile of bad queries: nothing to multiply
        }
        __syncwarp();
        named_sync(bX, kIssXN);  // layer 1's result converted (or the bad tile taken over)
        if (tdec < D) {
          if (lane == 0) {
            fence_after();
#pragma unroll
            for (uint32_t kq = 0; kq < H / 16; ++kq) umma_ta(tD, tH + 8 * kq, dW2 + 16 * kq, id_hidden, kq);
            umma_ta(tD, tOnes, dW2 + 16 * (H / 16), id_hidden, 1);  // + bias
            umma_commit(mbar);
          }
          ++l3;
        }
        __syncwarp();
        // the next tile, while layer 2's result is converted
        stop = k + NC < K ? prepare(k + NC, dec, swap) : 0;
        __syncwarp();
        if (tdec < D) named_sync(bZ, kIssZN);  // layer 1 of the next tile overwrites the accumulator
      }
    } else {
      for (uint32_t k = c; k < K; k += NC) {
        const uint32_t jc = k / NC, t = blockIdx.x + k * grid;
        uint32_t dec, start, len;
        iwalk.at(seg, tst, D, t, dec, start, len);
        named_sync(bT, kIssTN);
        if (stop_flag[2 * c + (jc & 1)]) break;
        if (dec >= D) continue;
        named_sync(bY, kIssYN);
        if (lane == 0) {  // the bias, then the K steps of the converted half
          fence_after();
          umma_ta(tO, tOnes, dW3 + 16 * (H / 16), id_out, 0);
#pragma unroll
          for (uint32_t kq = 0; kq < H / 32; ++kq) umma_ta(tO, tH + 8 * kq, dW3 + 16 * kq, id_out, 1);
        }
        issued = true;
        __syncwarp();
        named_sync(bZ, kIssZN);
        if (lane == 0) {
          fence_after();
#pragma unroll
          for (uint32_t kq = H / 32; kq < H / 16; ++kq) umma_ta(tO, tH + 8 * kq, dW3 + 16 * kq, id_out, 1);
          umma_commit(obar);
        }
        __syncwarp();
      }
    }
    if (lane == 0 && issued) {  // no MMA of this issuer is in flight when tensor memory is released
      umma_commit(fbar);
      wait(fbar, 0);
    }
    __syncwarp();
  }
  fence_before();
  __syncthreads();
  if (warp == 0) {
    fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(tmem_base), "r"(TC::alloc)
                 : "memory");
  }
}

template <int H, bool BF16, bool TRI, bool WRAP, int NP, int NC, int SC, bool DBG>
cudaError_t launch_tm_t(const Assets &A, const WeightImages &W, const Buckets &B, size_t n, void *out,
                        unsigned long long *err, unsigned int *status, int num_sms, cudaStream_t st,
                        ntc_debug_row *dbg) {
  using M = TmSmem<H, NC, SC>;
  const size_t smem = M::total;
  const bool c8 = W.out_dim <= 8;
  static PerDevice attr[2];
  auto set_attrs = [&](auto kernel) {
    return attr[c8].once([&]() {
      // as little shared memory as the kernel needs: the rest of the array is L1
      const int carve = (int)((smem * 100 + 232448 - 1) / 232448);
      cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (e == cudaSuccess) e = cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout, carve);
      return e;
    });
  };
  {
    const cudaError_t e = c8 ? set_attrs(k_decode_tm<H, BF16, TRI, WRAP, 8, NP, NC, SC, DBG>)
                             : set_attrs(k_decode_tm<H, BF16, TRI, WRAP, 16, NP, NC, SC, DBG>);
    if (e != cudaSuccess) return e;
  }
  const size_t max_tiles = (n + kTile - 1) / kTile + A.num_decoders + 1;
  size_t grid = (size_t)num_sms;
  if (grid > max_tiles) grid = max_tiles;
  // vector row stores need a base aligned to the row: 32 bytes (fp32) or 16 (fp16)
  const int vec_out = ((uintptr_t)out & (W.out_half ? 15 : 31)) == 0;
  const unsigned threads = (NP + NC) * 128 + (issuer_warp<H>() ? NC * 64 : 0);
  // launched as a programmatic dependent of the bucketing: its prologue overlaps
  // the end of k_place
  cudaError_t e;
  if (c8)
    e = launch_pdl(k_decode_tm<H, BF16, TRI, WRAP, 8, NP, NC, SC, DBG>, dim3((unsigned)grid), dim3(threads), smem, st,
                   A, W, B, out, err, status, vec_out, dbg);
  else
    e = launch_pdl(k_decode_tm<H, BF16, TRI, WRAP, 16, NP, NC, SC, DBG>, dim3((unsigned)grid), dim3(threads), smem, st,
                   A, W, B, out, err, status, vec_out, dbg);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

// Every (H, precision, trilinear, address mode) shape of the standard decode,
// dispatched at run time: 4 producer + 4 consumer warpgroups at H = 64, 4 + 2
// at H = 128 (tensor memory holds two 128-column accumulators).
template <bool DBG>
cudaError_t dispatch_tm(const Assets &A, const WeightImages &W, const Buckets &B, size_t n, void *out,
                        unsigned long long *err, unsigned int *status, bool bf16, int num_sms, cudaStream_t st,
                        ntc_debug_row *dbg) {
  const bool tri = A.num_mips > 1, wrap = A.address_mode == 0;
#define NTC_WS2(H, TRI, WRAP, NP, NC, SC)                                                                    \
  return bf16 ? launch_tm_t<H, true, TRI, WRAP, NP, NC, SC, DBG>(A, W, B, n, out, err, status, num_sms, st, dbg) \
              : launch_tm_t<H, false, TRI, WRAP, NP, NC, SC, DBG>(A, W, B, n, out, err, status, num_sms, st, dbg)
#define NTC_WS(H, TRI, NP, NC, SC)              \
  do {                                          \
    if (wrap) NTC_WS2(H, TRI, true, NP, NC, SC); \
    NTC_WS2(H, TRI, false, NP, NC, SC);          \
  } while (0)
  if (W.hidden == 64) {
    if (tri) NTC_WS(64, true, 4, 4, 1);
    NTC_WS(64, false, 4, 4, 1);
  }
  if (tri) NTC_WS(128, true, 4, 2, 2);
  NTC_WS(128, false, 4, 2, 2);
#undef NTC_WS
#undef NTC_WS2
}

}  // namespace ntc
