// CUDA-core kernels: the fp32 reference decode over bucketed tiles, the debug
// kernels (taps, features) and the packing of decoder weights into the images
// the tensor-core kernels read.
#include <math.h>

#include "ntc_internal.cuh"

namespace ntc {
namespace {

__device__ __forceinline__ void count_bad(bool bad, unsigned long long *err) {
  unsigned m = __ballot_sync(0xFFFFFFFFu, bad);
  if (m && (threadIdx.x & 31) == __ffs(m) - 1) atomicAdd(err, (unsigned long long)__popc(m));
}

// fp32 decode: one 128-thread CTA per tile, one query per thread, the tile's
// decoder in shared memory as fp32 (W1[H][16], b1, W2[H][H], b2, W3^T[H][CP],
// b3[CP]).  Tiles are split into contiguous ranges per CTA so a CTA rarely
// changes decoder.
template <int H, int CP>
__global__ void __launch_bounds__(kTile) k_decode_fp32(Assets A, WeightImages W, Buckets B,
                                                       float *out, unsigned long long *err) {
  extern __shared__ float4 smem4[];
  float *sw = reinterpret_cast<float *>(smem4);
  const float *W1 = sw, *b1 = W1 + H * 16, *W2 = b1 + H, *b2 = W2 + H * H, *W3t = b2 + H,
              *b3 = W3t + H * CP;
  const uint32_t D = A.num_decoders, C = W.out_dim;
  const uint32_t T = __ldg(B.meta);
  const bool copied = rows_copied(B, D);
  const uint32_t t0 = (uint32_t)((unsigned long long)T * blockIdx.x / gridDim.x);
  const uint32_t t1 = (uint32_t)((unsigned long long)T * (blockIdx.x + 1) / gridDim.x);
  const size_t img_floats = f32_image_floats(H, C);
  uint32_t cur = 0xFFFFFFFFu;
  for (uint32_t t = t0; t < t1; ++t) {
    uint32_t dec, start, len;
    tile_info(B.meta, D, t, dec, start, len);
    if (dec != cur && dec < D) {
      __syncthreads();
      const float4 *src = reinterpret_cast<const float4 *>(W.f32 + (size_t)dec * W.f32_stride);
      for (uint32_t i = threadIdx.x; i < img_floats / 4; i += blockDim.x) smem4[i] = __ldg(src + i);
      __syncthreads();
      cur = dec;
    }
    const uint32_t r = threadIdx.x;
    const bool valid = r < len;
    ntc_query q;
    uint32_t oi = 0;
    bool bad = false;
    if (valid) {
      bucket_row(B, copied, start + r, oi, q);
      bad = dec == D || query_bad(A, q);
    }
    count_bad(valid && bad, err);
    if (!valid) continue;
    float *o_row = out + (size_t)oi * C;
    if (bad) {
      for (uint32_t c = 0; c < C; ++c) o_row[c] = __int_as_float(0x7fc00000);
      continue;
    }
    float f[kInDim];
    query_features(A, q, f);
    float h1[H];
#pragma unroll
    for (int j = 0; j < H; ++j) {
      const float4 *w = reinterpret_cast<const float4 *>(W1 + j * 16);
      float acc = b1[j];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        float4 x = w[i];
        acc = fmaf(x.x, f[4 * i], acc);
        acc = fmaf(x.y, f[4 * i + 1], acc);
        acc = fmaf(x.z, f[4 * i + 2], acc);
        acc = fmaf(x.w, f[4 * i + 3], acc);
      }
      h1[j] = fmaxf(acc, 0.0f);
    }
    float o[CP];
#pragma unroll
    for (int c = 0; c < CP; ++c) o[c] = b3[c];
#pragma unroll 4
    for (int j = 0; j < H; ++j) {
      const float4 *w = reinterpret_cast<const float4 *>(W2 + j * H);
      float acc = b2[j];
#pragma unroll
      for (int i = 0; i < H / 4; ++i) {
        float4 x = w[i];
        acc = fmaf(x.x, h1[4 * i], acc);
        acc = fmaf(x.y, h1[4 * i + 1], acc);
        acc = fmaf(x.z, h1[4 * i + 2], acc);
        acc = fmaf(x.w, h1[4 * i + 3], acc);
      }
      const float h = fmaxf(acc, 0.0f);
      const float4 *w3 = reinterpret_cast<const float4 *>(W3t + j * CP);
#pragma unroll
      for (int i = 0; i < CP / 4; ++i) {
        float4 x = w3[i];
        o[4 * i] = fmaf(x.x, h, o[4 * i]);
        o[4 * i + 1] = fmaf(x.y, h, o[4 * i + 1]);
        o[4 * i + 2] = fmaf(x.z, h, o[4 * i + 2]);
        o[4 * i + 3] = fmaf(x.w, h, o[4 * i + 3]);
      }
    }
#pragma unroll
    for (int c = 0; c < CP; ++c)
      if (c < (int)C) o_row[c] = 1.0f / (1.0f + expf(-o[c]));
  }
}

__global__ void k_debug_taps(Assets A, const ntc_query *qs, size_t n, unsigned long long *idx,
                             float *w, float *t_out) {
  const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const ntc_query q = load_query(qs + i);
  const uint32_t L = A.num_levels;
  unsigned long long *I = idx + i * L * 8;
  float *Wt = w + i * L * 8;
  for (uint32_t e = 0; e < L * 8; ++e) {
    I[e] = ~0ull;
    Wt[e] = 0.0f;
  }
  t_out[i] = 0.0f;
  if (query_bad(A, q)) return;
  float t;
  const int lo = select_mip(q.lod, A.num_mips, t);
  t_out[i] = t;
  const GridDesc *g = A.grids + (size_t)q.set_id * L * A.num_mips;
  for (uint32_t k = 0; k < L; ++k) {
    unsigned long long ix[4];
    float wt[4];
    grid_taps(g[k * A.num_mips + lo], q.u, q.v, A.address_mode, ix, wt);
    for (int p = 0; p < 4; ++p) {
      I[k * 8 + p] = ix[p];
      Wt[k * 8 + p] = wt[p];
    }
    if (t > 0.0f) {
      grid_taps(g[k * A.num_mips + lo + 1], q.u, q.v, A.address_mode, ix, wt);
      for (int p = 0; p < 4; ++p) {
        I[k * 8 + 4 + p] = ix[p];
        Wt[k * 8 + 4 + p] = wt[p];
      }
    }
  }
}

// The MLP input of every query: the standard kernels' feature code for the
// standard input (2 levels x 8 channels), the general one otherwise.
__global__ void k_debug_features(Assets A, const ntc_query *qs, size_t n, float *f_out) {
  const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const ntc_query q = load_query(qs + i);
  const uint32_t in = A.num_levels * A.channels + 4 * A.pe_frequencies;
  const bool standard = A.num_levels == kLevels && A.channels == kChannels && A.pe_frequencies == 0;
  float f[kGenMaxIn];
  if (query_bad(A, q)) {
#pragma unroll
    for (int c = 0; c < kGenMaxIn; ++c) f[c] = __int_as_float(0x7fc00000);
  } else if (standard) {
    float s[kInDim];
    query_features(A, q, s);
#pragma unroll
    for (int c = 0; c < kGenMaxIn; ++c) f[c] = c < kInDim ? s[c] : 0.0f;
  } else {
    gen_features(A, A.grids, q, f);
  }
#pragma unroll
  for (int c = 0; c < kGenMaxIn; ++c)
    if (c < (int)in) f_out[i * in + c] = f[c];
}

template <typename T>
__device__ __forceinline__ uint16_t to_bits(float x);
template <>
__device__ __forceinline__ uint16_t to_bits<__half>(float x) {
  return __half_as_ushort(__float2half_rn(x));
}
template <>
__device__ __forceinline__ uint16_t to_bits<__nv_bfloat16>(float x) {
  return __bfloat16_as_ushort(__float2bfloat16_rn(x));
}

// One CTA per decoder: fp32 weights (W1,b1,W2,b2,W3,b3) -> mma image and fp32 image.
template <typename T>
__global__ void k_pack(const float *w32, uint32_t H, uint32_t C, uint8_t *mma, size_t mma_stride,
                       float *f32, size_t f32_stride) {
  const uint32_t d = blockIdx.x;
  const size_t P = (size_t)H * 17 + (size_t)H * (H + 1) + (size_t)C * (H + 1);
  const float *p = w32 + (size_t)d * P;
  const float *W1 = p, *b1 = W1 + H * 16, *W2 = b1 + H, *b2 = W2 + (size_t)H * H, *W3 = b2 + H,
              *b3 = W3 + (size_t)C * H;
  // mma image
  uint16_t *m = reinterpret_cast<uint16_t *>(mma + (size_t)d * mma_stride);
  uint16_t *W1p = m, *W2p = W1p + H * 24, *W3p = W2p + (size_t)H * (H + 8);
  float *bias = reinterpret_cast<float *>(W3p + 16 * (H + 8));
  for (uint32_t i = threadIdx.x; i < H * 24; i += blockDim.x) {
    uint32_t r = i / 24, c = i % 24;
    W1p[i] = c < 16 ? to_bits<T>(W1[r * 16 + c]) : 0;
  }
  for (uint32_t i = threadIdx.x; i < H * (H + 8); i += blockDim.x) {
    uint32_t r = i / (H + 8), c = i % (H + 8);
    W2p[i] = c < H ? to_bits<T>(W2[(size_t)r * H + c]) : 0;
  }
  for (uint32_t i = threadIdx.x; i < 16 * (H + 8); i += blockDim.x) {
    uint32_t r = i / (H + 8), c = i % (H + 8);
    W3p[i] = (r < C && c < H) ? to_bits<T>(W3[(size_t)r * H + c]) : 0;
  }
  for (uint32_t i = threadIdx.x; i < 2 * H + 16; i += blockDim.x)
    bias[i] = i < H ? b1[i] : (i < 2 * H ? b2[i - H] : (i - 2 * H < C ? b3[i - 2 * H] : 0.0f));
  // fp32 image
  const uint32_t CP = out_pad(C);
  float *f = f32 + (size_t)d * f32_stride;
  float *fW1 = f, *fb1 = fW1 + H * 16, *fW2 = fb1 + H, *fb2 = fW2 + (size_t)H * H, *fW3t = fb2 + H,
        *fb3 = fW3t + (size_t)H * CP;
  for (uint32_t i = threadIdx.x; i < H * 16; i += blockDim.x) fW1[i] = W1[i];
  for (uint32_t i = threadIdx.x; i < H; i += blockDim.x) {
    fb1[i] = b1[i];
    fb2[i] = b2[i];
  }
  for (uint32_t i = threadIdx.x; i < H * H; i += blockDim.x) fW2[i] = W2[i];
  for (uint32_t i = threadIdx.x; i < H * CP; i += blockDim.x) {
    uint32_t j = i / CP, c = i % CP;
    fW3t[i] = c < C ? W3[(size_t)c * H + j] : 0.0f;
  }
  for (uint32_t i = threadIdx.x; i < CP; i += blockDim.x) fb3[i] = i < C ? b3[i] : 0.0f;
}

template <int H, int CP>
cudaError_t launch_fp32_t(const Assets &A, const WeightImages &W, const Buckets &B, size_t n,
                          float *out, unsigned long long *err, int num_sms, cudaStream_t st) {
  const size_t smem = f32_image_floats(H, W.out_dim) * sizeof(float);
  static PerDevice occ_of;
  const int occ = occ_of.value([&]() {
    cudaFuncSetAttribute(k_decode_fp32<H, CP>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
    const int o = resident_ctas(k_decode_fp32<H, CP>, kTile, smem);
    return o < 1 ? 1 : o;
  });
  size_t max_tiles = (n + kTile - 1) / kTile + A.num_decoders + 1;
  size_t grid = (size_t)num_sms * occ;
  if (grid > max_tiles) grid = max_tiles;
  k_decode_fp32<H, CP><<<(unsigned)grid, kTile, smem, st>>>(A, W, B, out, err);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_decode_fp32(const Assets &A, const WeightImages &W, const Buckets &B, size_t n,
                               float *out, unsigned long long *err, int num_sms, cudaStream_t st,
                               int *launches) {
  *launches += 1;
  const bool c8 = W.out_dim <= 8;
  if (W.hidden == 64)
    return c8 ? launch_fp32_t<64, 8>(A, W, B, n, out, err, num_sms, st)
              : launch_fp32_t<64, 16>(A, W, B, n, out, err, num_sms, st);
  return c8 ? launch_fp32_t<128, 8>(A, W, B, n, out, err, num_sms, st)
            : launch_fp32_t<128, 16>(A, W, B, n, out, err, num_sms, st);
}

cudaError_t launch_debug_taps(const Assets &A, const ntc_query *q, size_t n, unsigned long long *idx,
                              float *w, float *t, cudaStream_t st, int *launches) {
  *launches += 1;
  k_debug_taps<<<(unsigned)((n + 127) / 128), 128, 0, st>>>(A, q, n, idx, w, t);
  return cudaGetLastError();
}

cudaError_t launch_debug_features(const Assets &A, const ntc_query *q, size_t n, float *f,
                                  cudaStream_t st, int *launches) {
  *launches += 1;
  k_debug_features<<<(unsigned)((n + 127) / 128), 128, 0, st>>>(A, q, n, f);
  return cudaGetLastError();
}

cudaError_t launch_pack_weights(const float *w32, uint32_t D, uint32_t H, uint32_t C, bool bf16,
                                uint8_t *mma, size_t mma_stride, float *f32, size_t f32_stride,
                                uint8_t *tc, size_t tc_stride, cudaStream_t st) {
  if (bf16)
    k_pack<__nv_bfloat16><<<D, 256, 0, st>>>(w32, H, C, mma, mma_stride, f32, f32_stride);
  else
    k_pack<__half><<<D, 256, 0, st>>>(w32, H, C, mma, mma_stride, f32, f32_stride);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  return launch_pack_tc(w32, D, H, C, bf16, tc, tc_stride, st);
}

}  // namespace ntc
