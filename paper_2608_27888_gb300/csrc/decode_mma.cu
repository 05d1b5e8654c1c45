// Warp-level tensor-core decode (mma.sync m16n8k16, fp16/bf16 operands, fp32
// accumulation).  Two users:
//   k_decode_mma        bucketed: a 128-thread CTA decodes one single-decoder
//                       128-query tile, each warp 32 rows; the decoder's
//                       weights sit in shared memory and are read with ldmatrix
//   k_decode_divergent  unsorted: each warp takes 32 consecutive queries and
//                       loops over its distinct decoders, evaluating each one
//                       on the whole warp with the other rows masked -- the
//                       non-shared setting of Sec. 4.4 (Tables 5-6), where the
//                       cost grows with the decoders per warp
// The hidden activations never leave registers: the fp32 accumulator fragment
// of one layer, after bias (preloaded into the accumulator) and ReLU, is
// repacked as the A fragment of the next layer.
#include "ntc_internal.cuh"

namespace ntc {
namespace {

constexpr int kFeatStride = 24;  // halves per staged feature row (16 + 8 pad)

template <bool BF16>
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
  if (BF16)
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
        "{%8,%9}, {%0,%1,%2,%3};\n"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
  else
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
        "{%8,%9}, {%0,%1,%2,%3};\n"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Two fp32 values -> packed 16-bit pair (lo in the low half), optional ReLU.
template <bool BF16, bool RELU>
__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
  uint32_t r;
  if (BF16) {
    if (RELU) asm("cvt.rn.relu.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    else asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  } else {
    if (RELU) asm("cvt.rn.relu.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    else asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  }
  return r;
}

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2,
                                        uint32_t &r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

// B fragments of a weight matrix stored [n][k] with `stride` elements per row.
// frag(nt, kt) = {W[nt*8+g][kt*16+2tq .. +1], W[nt*8+g][kt*16+8+2tq .. +1]}.
struct SmemB {
  uint32_t base;  // shared address of W[0][0]
  int stride;     // elements per row
  // fragments of n-tiles nt0, nt0+1 at k-tile kt
  __device__ __forceinline__ void pair(int nt0, int kt, uint32_t (&b)[2][2]) const {
    const int lane = threadIdx.x & 31;
    const int j = lane >> 3;  // which 8x8 matrix this lane addresses
    const int row = (nt0 + (j >> 1)) * 8 + (lane & 7);
    const int col = kt * 16 + (j & 1) * 8;
    ldsm_x4(base + (uint32_t)(row * stride + col) * 2u, b[0][0], b[0][1], b[1][0], b[1][1]);
  }
  // fragments of n-tile nt at k-tiles kt0, kt0+1
  __device__ __forceinline__ void ktwo(int nt, int kt0, uint32_t (&b)[2][2]) const {
    const int lane = threadIdx.x & 31;
    const int j = lane >> 3;
    const int row = nt * 8 + (lane & 7);
    const int col = (kt0 + (j >> 1)) * 16 + (j & 1) * 8;
    ldsm_x4(base + (uint32_t)(row * stride + col) * 2u, b[0][0], b[0][1], b[1][0], b[1][1]);
  }
};

struct GlobalB {
  const uint16_t *base;
  int stride;
  __device__ __forceinline__ uint32_t ld(int n, int k) const {
    return __ldg(reinterpret_cast<const uint32_t *>(base + (size_t)n * stride + k));
  }
  __device__ __forceinline__ void pair(int nt0, int kt, uint32_t (&b)[2][2]) const {
    const int lane = threadIdx.x & 31, g = lane >> 2, tq = lane & 3;
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      b[i][0] = ld((nt0 + i) * 8 + g, kt * 16 + 2 * tq);
      b[i][1] = ld((nt0 + i) * 8 + g, kt * 16 + 8 + 2 * tq);
    }
  }
  __device__ __forceinline__ void ktwo(int nt, int kt0, uint32_t (&b)[2][2]) const {
    const int lane = threadIdx.x & 31, g = lane >> 2, tq = lane & 3;
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      b[i][0] = ld(nt * 8 + g, (kt0 + i) * 16 + 2 * tq);
      b[i][1] = ld(nt * 8 + g, (kt0 + i) * 16 + 8 + 2 * tq);
    }
  }
};

// The 3-layer MLP on 32 rows (two m16 tiles) of one warp.
//   a1[m]    layer-1 A fragments (features, K = 16)
//   o[m][n]  output accumulators (bias b3 included), n-tiles of 8 columns
//   live[m]  false skips m-tile m (no row of it needs this decoder)
template <int H, int NT3, bool BF16, class BL>
__device__ __forceinline__ void warp_mlp(const uint32_t (&a1)[2][4], const BL &W1, const BL &W2,
                                         const BL &W3, const float *b1, const float *b2,
                                         const float *b3, const bool (&live)[2],
                                         float (&o)[2][NT3][4]) {
  const int lane = threadIdx.x & 31, tq = lane & 3;
  constexpr int KT = H / 16;  // k-tiles of the hidden layers
  // layer 1 -> h1 as A fragments
  uint32_t h1[2][KT][4];
#pragma unroll
  for (int kt = 0; kt < KT; ++kt) {
    uint32_t b[2][2];
    W1.pair(2 * kt, 0, b);
    float acc[2][2][4];
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const float2 bb = *reinterpret_cast<const float2 *>(b1 + (2 * kt + i) * 8 + 2 * tq);
#pragma unroll
      for (int m = 0; m < 2; ++m) {
        acc[m][i][0] = bb.x;
        acc[m][i][1] = bb.y;
        acc[m][i][2] = bb.x;
        acc[m][i][3] = bb.y;
      }
    }
#pragma unroll
    for (int m = 0; m < 2; ++m)
      if (live[m]) {
        mma16816<BF16>(acc[m][0], a1[m], b[0][0], b[0][1]);
        mma16816<BF16>(acc[m][1], a1[m], b[1][0], b[1][1]);
      }
#pragma unroll
    for (int m = 0; m < 2; ++m) {
      h1[m][kt][0] = pack2<BF16, true>(acc[m][0][0], acc[m][0][1]);
      h1[m][kt][1] = pack2<BF16, true>(acc[m][0][2], acc[m][0][3]);
      h1[m][kt][2] = pack2<BF16, true>(acc[m][1][0], acc[m][1][1]);
      h1[m][kt][3] = pack2<BF16, true>(acc[m][1][2], acc[m][1][3]);
    }
  }
  // output accumulators start at b3
#pragma unroll
  for (int n = 0; n < NT3; ++n) {
    const float2 bb = *reinterpret_cast<const float2 *>(b3 + n * 8 + 2 * tq);
#pragma unroll
    for (int m = 0; m < 2; ++m) {
      o[m][n][0] = bb.x;
      o[m][n][1] = bb.y;
      o[m][n][2] = bb.x;
      o[m][n][3] = bb.y;
    }
  }
  // layer 2, 16 output columns at a time; each slice is immediately the A
  // fragment of one k-tile of layer 3
#pragma unroll
  for (int s = 0; s < KT; ++s) {
    float acc[2][2][4];
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const float2 bb = *reinterpret_cast<const float2 *>(b2 + (2 * s + i) * 8 + 2 * tq);
#pragma unroll
      for (int m = 0; m < 2; ++m) {
        acc[m][i][0] = bb.x;
        acc[m][i][1] = bb.y;
        acc[m][i][2] = bb.x;
        acc[m][i][3] = bb.y;
      }
    }
#pragma unroll
    for (int kt = 0; kt < KT; ++kt) {
      uint32_t b[2][2];
      W2.pair(2 * s, kt, b);
#pragma unroll
      for (int m = 0; m < 2; ++m)
        if (live[m]) {
          mma16816<BF16>(acc[m][0], h1[m][kt], b[0][0], b[0][1]);
          mma16816<BF16>(acc[m][1], h1[m][kt], b[1][0], b[1][1]);
        }
    }
    uint32_t a3[2][4];
#pragma unroll
    for (int m = 0; m < 2; ++m) {
      a3[m][0] = pack2<BF16, true>(acc[m][0][0], acc[m][0][1]);
      a3[m][1] = pack2<BF16, true>(acc[m][0][2], acc[m][0][3]);
      a3[m][2] = pack2<BF16, true>(acc[m][1][0], acc[m][1][1]);
      a3[m][3] = pack2<BF16, true>(acc[m][1][2], acc[m][1][3]);
    }
#pragma unroll
    for (int n = 0; n < NT3; ++n) {
      uint32_t b[2][2];
      // k-tile s of W3, n-tile n (the second half of ktwo is unused when s is
      // the last k-tile; load k-tiles in pairs and use the matching one)
      W3.ktwo(n, s & ~1, b);
      const int which = s & 1;
#pragma unroll
      for (int m = 0; m < 2; ++m)
        if (live[m]) mma16816<BF16>(o[m][n], a3[m], b[which][0], b[which][1]);
    }
  }
}

__device__ __forceinline__ float sigmoidf_fast(float x) { return 1.0f / (1.0f + __expf(-x)); }

// Stage one feature row per lane into shared memory, then read the A
// fragments of both m-tiles with ldmatrix.
template <bool BF16>
__device__ __forceinline__ void features_to_afrag(const float (&f)[kInDim], uint16_t *stage,
                                                  uint32_t (&a1)[2][4]) {
  const int lane = threadIdx.x & 31;
  uint4 lo, hi;
  lo.x = pack2<BF16, false>(f[0], f[1]);
  lo.y = pack2<BF16, false>(f[2], f[3]);
  lo.z = pack2<BF16, false>(f[4], f[5]);
  lo.w = pack2<BF16, false>(f[6], f[7]);
  hi.x = pack2<BF16, false>(f[8], f[9]);
  hi.y = pack2<BF16, false>(f[10], f[11]);
  hi.z = pack2<BF16, false>(f[12], f[13]);
  hi.w = pack2<BF16, false>(f[14], f[15]);
  uint4 *row = reinterpret_cast<uint4 *>(stage + lane * kFeatStride);
  row[0] = lo;
  row[1] = hi;
  __syncwarp();
#pragma unroll
  for (int m = 0; m < 2; ++m) {
    const int j = lane >> 3;
    const int r = m * 16 + (lane & 7) + (j & 1) * 8;
    const int c = (j >> 1) * 8;
    ldsm_x4(smem_u32(stage + r * kFeatStride + c), a1[m][0], a1[m][1], a1[m][2], a1[m][3]);
  }
  __syncwarp();
}

// Write the output fragment rows of one warp: row = m*16 + g (+8), columns
// n*8 + 2tq (+1); `rowmask` bit r set = row r of the warp is written.
template <int NT3>
__device__ __forceinline__ void store_out(const float (&o)[2][NT3][4], uint32_t rowmask,
                                          const uint32_t *orig_rows, float *out, uint32_t C) {
  const int lane = threadIdx.x & 31, g = lane >> 2, tq = lane & 3;
#pragma unroll
  for (int m = 0; m < 2; ++m)
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int r = m * 16 + g + 8 * h;
      if (!((rowmask >> r) & 1u)) continue;
      float *dst = out + (size_t)orig_rows[r] * C;
#pragma unroll
      for (int n = 0; n < NT3; ++n) {
        const uint32_t c = n * 8 + 2 * tq;
        if (c < C) dst[c] = sigmoidf_fast(o[m][n][2 * h]);
        if (c + 1 < C) dst[c + 1] = sigmoidf_fast(o[m][n][2 * h + 1]);
      }
    }
}

template <int H>
struct MmaImage {
  static constexpr int s1 = 24, s2 = H + 8, s3 = H + 8;
  static constexpr int off_w2 = H * s1;              // elements
  static constexpr int off_w3 = off_w2 + H * s2;
  static constexpr int off_bias = off_w3 + 16 * s3;  // elements (bias as fp32 after)
  static constexpr size_t bytes = (size_t)off_bias * 2 + (size_t)(2 * H + 16) * 4;
};

template <int H, int NT3, bool BF16>
__global__ void __launch_bounds__(kTile) k_decode_mma(Assets A, WeightImages W, Buckets B,
                                                      float *out, unsigned long long *err) {
  using I = MmaImage<H>;
  extern __shared__ uint4 smem[];
  uint16_t *sw = reinterpret_cast<uint16_t *>(smem);
  const float *sb = reinterpret_cast<const float *>(sw + I::off_bias);
  uint16_t *stage_all = reinterpret_cast<uint16_t *>(reinterpret_cast<uint8_t *>(smem) + ((I::bytes + 15) & ~(size_t)15));
  __shared__ uint32_t orig[kTile];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint16_t *stage = stage_all + warp * 32 * kFeatStride;
  const uint32_t D = A.num_decoders, C = W.out_dim;
  const uint32_t T = __ldg(B.meta);
  const bool copied = rows_copied(B, D);
  const uint32_t t0 = (uint32_t)((unsigned long long)T * blockIdx.x / gridDim.x);
  const uint32_t t1 = (uint32_t)((unsigned long long)T * (blockIdx.x + 1) / gridDim.x);
  const SmemB W1{smem_u32(sw), I::s1}, W2{smem_u32(sw + I::off_w2), I::s2},
      W3{smem_u32(sw + I::off_w3), I::s3};
  const uint32_t img16 = (uint32_t)((I::bytes + 15) / 16);
  uint32_t cur = 0xFFFFFFFFu;
  for (uint32_t t = t0; t < t1; ++t) {
    uint32_t dec, start, len;
    tile_info(B.meta, D, t, dec, start, len);
    if (dec != cur && dec < D) {
      __syncthreads();
      const uint4 *src = reinterpret_cast<const uint4 *>(W.mma + (size_t)dec * W.mma_stride);
      for (uint32_t i = threadIdx.x; i < img16; i += blockDim.x) smem[i] = __ldg(src + i);
      __syncthreads();
      cur = dec;
    }
    const uint32_t r = warp * 32 + lane;
    const bool valid = r < len;
    ntc_query q;
    bool bad = false;
    uint32_t oi = 0;
    if (valid) {
      bucket_row(B, copied, start + r, oi, q);
      bad = dec == D || query_bad(A, q);
    }
    orig[r] = oi;
    const uint32_t badm = __ballot_sync(0xFFFFFFFFu, valid && bad);
    if (badm && lane == __ffs(badm) - 1) atomicAdd(err, (unsigned long long)__popc(badm));
    if (valid && bad)
      for (uint32_t c = 0; c < C; ++c) out[(size_t)oi * C + c] = __int_as_float(0x7fc00000);
    const uint32_t goodm = __ballot_sync(0xFFFFFFFFu, valid && !bad);
    if (goodm == 0) continue;  // warp-uniform
    float f[kInDim];
    if (valid && !bad) query_features(A, q, f);
    else
#pragma unroll
      for (int c = 0; c < kInDim; ++c) f[c] = 0.0f;
    uint32_t a1[2][4];
    features_to_afrag<BF16>(f, stage, a1);
    const bool live[2] = {(goodm & 0xFFFFu) != 0, (goodm >> 16) != 0};
    float o[2][NT3][4];
    warp_mlp<H, NT3, BF16>(a1, W1, W2, W3, sb, sb + H, sb + 2 * H, live, o);
    __syncwarp();
    store_out<NT3>(o, goodm, orig + warp * 32, out, C);
  }
}

// At most 128 registers a thread, so that four CTAs (16 warps) fit on an SM.
// The warp MLP wants ~180 at H = 128 (both m-tiles of the hidden layer as A
// fragments); the few spills cost less than the latency that eight warps
// cannot hide (measured on config 5: 13.8 -> 11.2 ms; 3 CTAs: 14.0, 5: 18.2).
template <int H, int NT3, bool BF16>
__global__ void __launch_bounds__(128, 4) k_decode_divergent(Assets A, WeightImages W,
                                                          const ntc_query *qs, size_t n,
                                                          float *out, unsigned long long *err) {
  using I = MmaImage<H>;
  __shared__ __align__(16) uint16_t stage_all[4 * 32 * kFeatStride];
  __shared__ uint32_t orig_all[128];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint16_t *stage = stage_all + warp * 32 * kFeatStride;
  uint32_t *orig = orig_all + warp * 32;
  const uint32_t C = W.out_dim;
  const size_t nwarps = (n + 31) / 32;
  for (size_t w = (size_t)blockIdx.x * 4 + warp; w < nwarps; w += (size_t)gridDim.x * 4) {
    const size_t i = w * 32 + lane;
    const bool valid = i < n;
    ntc_query q;
    bool bad = false;
    if (valid) {
      q = load_query(qs + i);
      bad = query_bad(A, q);
    }
    orig[lane] = (uint32_t)i;
    const uint32_t badm = __ballot_sync(0xFFFFFFFFu, valid && bad);
    if (badm && lane == __ffs(badm) - 1) atomicAdd(err, (unsigned long long)__popc(badm));
    if (valid && bad)
      for (uint32_t c = 0; c < C; ++c) out[i * C + c] = __int_as_float(0x7fc00000);
    const bool good = valid && !bad;
    uint32_t pending = __ballot_sync(0xFFFFFFFFu, good);
    if (pending == 0) continue;
    float f[kInDim];
    if (good) query_features(A, q, f);
    else
#pragma unroll
      for (int c = 0; c < kInDim; ++c) f[c] = 0.0f;
    uint32_t a1[2][4];
    features_to_afrag<BF16>(f, stage, a1);
    const uint32_t mydec = good ? __ldg(A.map + q.set_id) : 0xFFFFFFFFu;
    while (pending) {
      const uint32_t d = __shfl_sync(0xFFFFFFFFu, mydec, __ffs(pending) - 1);
      const uint32_t active = __ballot_sync(0xFFFFFFFFu, mydec == d);
      const uint16_t *img = reinterpret_cast<const uint16_t *>(W.mma + (size_t)d * W.mma_stride);
      const GlobalB W1{img, I::s1}, W2{img + I::off_w2, I::s2}, W3{img + I::off_w3, I::s3};
      const float *bias = reinterpret_cast<const float *>(img + I::off_bias);
      const bool live[2] = {(active & 0xFFFFu) != 0, (active >> 16) != 0};
      float o[2][NT3][4];
      warp_mlp<H, NT3, BF16>(a1, W1, W2, W3, bias, bias + H, bias + 2 * H, live, o);
      store_out<NT3>(o, active, orig, out, C);
      pending &= ~active;
    }
    __syncwarp();
  }
}

template <int H, int NT3, bool BF16>
cudaError_t launch_mma_t(const Assets &A, const WeightImages &W, const Buckets &B, size_t n,
                         float *out, unsigned long long *err, int num_sms, cudaStream_t st) {
  using I = MmaImage<H>;
  const size_t smem = ((I::bytes + 15) & ~(size_t)15) + (size_t)4 * 32 * kFeatStride * 2;
  static PerDevice occ_of;
  const int occ = occ_of.value([&]() {
    cudaFuncSetAttribute(k_decode_mma<H, NT3, BF16>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
    const int o = resident_ctas(k_decode_mma<H, NT3, BF16>, kTile, smem);
    return o < 1 ? 1 : o;
  });
  size_t max_tiles = (n + kTile - 1) / kTile + A.num_decoders + 1;
  size_t grid = (size_t)num_sms * occ;
  if (grid > max_tiles) grid = max_tiles;
  k_decode_mma<H, NT3, BF16><<<(unsigned)grid, kTile, smem, st>>>(A, W, B, out, err);
  return cudaGetLastError();
}

template <int H, int NT3, bool BF16>
cudaError_t launch_div_t(const Assets &A, const WeightImages &W, const ntc_query *q, size_t n,
                         float *out, unsigned long long *err, int num_sms, cudaStream_t st) {
  static PerDevice occ_of;
  const int occ = occ_of.value([&]() {
    const int o = resident_ctas(k_decode_divergent<H, NT3, BF16>, 128, 0);
    return o < 1 ? 1 : o;
  });
  size_t blocks = (n + 127) / 128;
  size_t grid = (size_t)num_sms * occ * 4;
  if (grid > blocks) grid = blocks;
  k_decode_divergent<H, NT3, BF16><<<(unsigned)grid, 128, 0, st>>>(A, W, q, n, out, err);
  return cudaGetLastError();
}

}  // namespace

#define NTC_DISPATCH(FN, ...)                                                        \
  do {                                                                               \
    const bool c8 = W.out_dim <= 8;                                                  \
    if (W.hidden == 64) {                                                            \
      if (bf16) return c8 ? FN<64, 1, true>(__VA_ARGS__) : FN<64, 2, true>(__VA_ARGS__);   \
      return c8 ? FN<64, 1, false>(__VA_ARGS__) : FN<64, 2, false>(__VA_ARGS__);           \
    }                                                                                \
    if (bf16) return c8 ? FN<128, 1, true>(__VA_ARGS__) : FN<128, 2, true>(__VA_ARGS__);   \
    return c8 ? FN<128, 1, false>(__VA_ARGS__) : FN<128, 2, false>(__VA_ARGS__);           \
  } while (0)

cudaError_t launch_decode_mma(const Assets &A, const WeightImages &W, const Buckets &B, size_t n,
                              float *out, unsigned long long *err, bool bf16, int num_sms,
                              cudaStream_t st, int *launches) {
  *launches += 1;
  NTC_DISPATCH(launch_mma_t, A, W, B, n, out, err, num_sms, st);
}

cudaError_t launch_decode_divergent(const Assets &A, const WeightImages &W, const ntc_query *q,
                                    size_t n, float *out, unsigned long long *err, bool bf16,
                                    int num_sms, cudaStream_t st, int *launches) {
  *launches += 1;
  NTC_DISPATCH(launch_div_t, A, W, q, n, out, err, num_sms, st);
}

}  // namespace ntc
