// Per-lane FMA decode without sorting: the in-run analogue of the paper's
// "Non-Shared FMA" kernel (Sec. 4.4, Tables 5-6).
//
// Every thread takes one query in its original order and evaluates that
// query's decoder on its own with fp32 fused multiply-adds (two lanes of fp32
// per instruction), reading the decoder's weights through the L1 cache.  No
// thread waits for another: a warp whose 32 queries need d distinct decoders
// issues the same instruction stream as a warp with one decoder, but every
// weight load touches d different cache lines instead of one.  That memory
// divergence, not control flow, is what the shared decoder removes here.
//
// Operands follow the context's precision: with a tensor-core precision the
// features, the weights and the hidden activations are rounded to fp16/bf16 as
// the tensor-core kernels round them (fp32 accumulation and biases); with FP32
// nothing is rounded.
#include <math.h>

#include "ntc_internal.cuh"

namespace ntc {
namespace {

template <typename T>
struct Elem;

template <>
struct Elem<float> {
  static __device__ __forceinline__ void load8(const float *p, float (&w)[8]) {
    const float4 a = __ldg(reinterpret_cast<const float4 *>(p));
    const float4 b = __ldg(reinterpret_cast<const float4 *>(p) + 1);
    w[0] = a.x, w[1] = a.y, w[2] = a.z, w[3] = a.w;
    w[4] = b.x, w[5] = b.y, w[6] = b.z, w[7] = b.w;
  }
  static __device__ __forceinline__ float round(float x) { return x; }
  static __device__ __forceinline__ float cvt(float x) { return x; }
};

template <>
struct Elem<__half> {
  static __device__ __forceinline__ void load8(const __half *p, float (&w)[8]) {
    const uint4 r = __ldg(reinterpret_cast<const uint4 *>(p));
    const __half2 *h = reinterpret_cast<const __half2 *>(&r);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 x = __half22float2(h[i]);
      w[2 * i] = x.x, w[2 * i + 1] = x.y;
    }
  }
  static __device__ __forceinline__ float round(float x) { return __half2float(__float2half_rn(x)); }
  static __device__ __forceinline__ __half cvt(float x) { return __float2half_rn(x); }
};

template <>
struct Elem<__nv_bfloat16> {
  static __device__ __forceinline__ void load8(const __nv_bfloat16 *p, float (&w)[8]) {
    const uint4 r = __ldg(reinterpret_cast<const uint4 *>(p));
    const __nv_bfloat162 *h = reinterpret_cast<const __nv_bfloat162 *>(&r);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 x = __bfloat1622float2(h[i]);
      w[2 * i] = x.x, w[2 * i + 1] = x.y;
    }
  }
  static __device__ __forceinline__ float round(float x) {
    return __bfloat162float(__float2bfloat16_rn(x));
  }
  static __device__ __forceinline__ __nv_bfloat16 cvt(float x) { return __float2bfloat16_rn(x); }
};

__device__ __forceinline__ void count_bad_warp(bool bad, unsigned long long *err) {
  const unsigned m = __ballot_sync(0xFFFFFFFFu, bad);
  if (m && (threadIdx.x & 31) == __ffs(m) - 1) atomicAdd(err, (unsigned long long)__popc(m));
}

// acc += (w[0..7] . x[0..7]) as four packed fp32 pairs
__device__ __forceinline__ float2 dot8(const float (&w)[8], const float *x, float2 acc) {
#pragma unroll
  for (int p = 0; p < 4; ++p)
    acc = __ffma2_rn(make_float2(w[2 * p], w[2 * p + 1]), make_float2(x[2 * p], x[2 * p + 1]), acc);
  return acc;
}

// Register cap: each lane holds its whole hidden vector, so the compiler takes
// ~230 registers a thread at H = 128 (2 CTAs, 8 warps per SM) and ~140 at
// H = 64.  Capping them for 4 (H = 128) or 3 (H = 64) CTAs per SM spills a
// little and hides more of the gather latency; measured on config 5 158 -> 97
// ms, on the 1080p G-buffer (H = 64) 1.24 -> 1.09 ms; more CTAs were slower.
template <int H, int CP, typename T>
__global__ void __launch_bounds__(128, H >= 128 ? 4 : 3) k_decode_divergent_fma(Assets A, const uint8_t *img, size_t stride,
                                                              uint32_t C, const ntc_query *qs, size_t n,
                                                              float *out, unsigned long long *err) {
  using E = Elem<T>;
  const size_t step = (size_t)gridDim.x * blockDim.x;
  const size_t nr = (n + 31) & ~(size_t)31;  // whole warps iterate together
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < nr; i += step) {
    const bool valid = i < n;
    ntc_query q;
    bool bad = false;
    if (valid) {
      q = load_query(qs + i);
      bad = query_bad(A, q);
    }
    count_bad_warp(valid && bad, err);
    if (!valid) continue;
    float *o_row = out + i * C;
    if (bad) {
      for (uint32_t c = 0; c < C; ++c) o_row[c] = __int_as_float(0x7fc00000);
      continue;
    }
    const uint32_t dec = __ldg(A.map + q.set_id);
    const T *W1 = reinterpret_cast<const T *>(img + (size_t)dec * stride);
    const T *W2 = W1 + H * 16, *W3t = W2 + H * H;
    const float *b1 = reinterpret_cast<const float *>(W3t + H * CP), *b2 = b1 + H, *b3 = b2 + H;
    float f[kInDim];
    query_features(A, q, f);
#pragma unroll
    for (int c = 0; c < kInDim; ++c) f[c] = E::round(f[c]);
    float h1[H];
#pragma unroll
    for (int j = 0; j < H; ++j) {
      float w[8];
      E::load8(W1 + j * 16, w);
      float2 acc = dot8(w, f, make_float2(0.0f, 0.0f));
      E::load8(W1 + j * 16 + 8, w);
      acc = dot8(w, f + 8, acc);
      h1[j] = E::round(fmaxf(__fadd_rn(__fadd_rn(acc.x, acc.y), __ldg(b1 + j)), 0.0f));
    }
    float o[CP];
#pragma unroll
    for (int c = 0; c < CP; ++c) o[c] = 0.0f;
#pragma unroll 2
    for (int j = 0; j < H; ++j) {
      float2 acc = make_float2(0.0f, 0.0f);
#pragma unroll
      for (int i0 = 0; i0 < H; i0 += 8) {
        float w[8];
        E::load8(W2 + j * H + i0, w);
        acc = dot8(w, h1 + i0, acc);
      }
      const float h = E::round(fmaxf(__fadd_rn(__fadd_rn(acc.x, acc.y), __ldg(b2 + j)), 0.0f));
#pragma unroll
      for (int c0 = 0; c0 < CP; c0 += 8) {
        float w[8];
        E::load8(W3t + j * CP + c0, w);
#pragma unroll
        for (int p = 0; p < 8; ++p) o[c0 + p] = fmaf(w[p], h, o[c0 + p]);
      }
    }
#pragma unroll
    for (int c = 0; c < CP; ++c)
      if (c < (int)C) o_row[c] = 1.0f / (1.0f + expf(-__fadd_rn(o[c], __ldg(b3 + c))));
  }
}

// One CTA per decoder: fp32 weights (W1,b1,W2,b2,W3,b3) -> the FMA image.
template <typename T>
__global__ void k_pack_fma(const float *w32, uint32_t H, uint32_t C, uint8_t *img, size_t stride) {
  using E = Elem<T>;
  const uint32_t d = blockIdx.x, CP = out_pad(C);
  const size_t P = (size_t)H * 17 + (size_t)H * (H + 1) + (size_t)C * (H + 1);
  const float *p = w32 + (size_t)d * P;
  const float *W1 = p, *b1 = W1 + H * 16, *W2 = b1 + H, *b2 = W2 + (size_t)H * H, *W3 = b2 + H,
              *b3 = W3 + (size_t)C * H;
  T *oW1 = reinterpret_cast<T *>(img + (size_t)d * stride);
  T *oW2 = oW1 + H * 16, *oW3t = oW2 + (size_t)H * H;
  float *ob = reinterpret_cast<float *>(oW3t + (size_t)H * CP);
  for (uint32_t i = threadIdx.x; i < H * 16; i += blockDim.x) oW1[i] = E::cvt(W1[i]);
  for (uint32_t i = threadIdx.x; i < H * H; i += blockDim.x) oW2[i] = E::cvt(W2[i]);
  for (uint32_t i = threadIdx.x; i < H * CP; i += blockDim.x) {
    const uint32_t j = i / CP, c = i % CP;
    oW3t[i] = E::cvt(c < C ? W3[(size_t)c * H + j] : 0.0f);
  }
  for (uint32_t i = threadIdx.x; i < 2 * H + CP; i += blockDim.x)
    ob[i] = i < H ? b1[i] : (i < 2 * H ? b2[i - H] : (i - 2 * H < C ? b3[i - 2 * H] : 0.0f));
}

template <int H, int CP, typename T>
cudaError_t launch_fma_t(const Assets &A, const WeightImages &W, const ntc_query *q, size_t n, float *out,
                         unsigned long long *err, int num_sms, cudaStream_t st) {
  static PerDevice occ_of;
  const int occ = occ_of.value([&]() {
    const int o = resident_ctas(k_decode_divergent_fma<H, CP, T>, 128, 0);
    return o < 1 ? 1 : o;
  });
  const size_t blocks = (n + 127) / 128;
  size_t grid = (size_t)num_sms * occ * 8;
  if (grid > blocks) grid = blocks;
  k_decode_divergent_fma<H, CP, T><<<(unsigned)grid, 128, 0, st>>>(A, W.fma, W.fma_stride, W.out_dim, q, n,
                                                                    out, err);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_fma_h(const Assets &A, const WeightImages &W, const ntc_query *q, size_t n, float *out,
                         unsigned long long *err, int num_sms, cudaStream_t st) {
  const bool c8 = W.out_dim <= 8;
  if (W.hidden == 64)
    return c8 ? launch_fma_t<64, 8, T>(A, W, q, n, out, err, num_sms, st)
              : launch_fma_t<64, 16, T>(A, W, q, n, out, err, num_sms, st);
  return c8 ? launch_fma_t<128, 8, T>(A, W, q, n, out, err, num_sms, st)
            : launch_fma_t<128, 16, T>(A, W, q, n, out, err, num_sms, st);
}

}  // namespace

cudaError_t launch_decode_divergent_fma(const Assets &A, const WeightImages &W, const ntc_query *q, size_t n,
                                        float *out, unsigned long long *err, ntc_precision prec, int num_sms,
                                        cudaStream_t st, int *launches) {
  *launches += 1;
  if (prec == NTC_PREC_FP32) return launch_fma_h<float>(A, W, q, n, out, err, num_sms, st);
  if (prec == NTC_PREC_TC_BF16) return launch_fma_h<__nv_bfloat16>(A, W, q, n, out, err, num_sms, st);
  return launch_fma_h<__half>(A, W, q, n, out, err, num_sms, st);
}

cudaError_t launch_pack_fma(const float *w32, uint32_t D, uint32_t H, uint32_t C, ntc_precision prec,
                            uint8_t *fma, size_t fma_stride, cudaStream_t st) {
  if (prec == NTC_PREC_FP32)
    k_pack_fma<float><<<D, 256, 0, st>>>(w32, H, C, fma, fma_stride);
  else if (prec == NTC_PREC_TC_BF16)
    k_pack_fma<__nv_bfloat16><<<D, 256, 0, st>>>(w32, H, C, fma, fma_stride);
  else
    k_pack_fma<__half><<<D, 256, 0, st>>>(w32, H, C, fma, fma_stride);
  return cudaGetLastError();
}

}  // namespace ntc
