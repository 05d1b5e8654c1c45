// tcgen05 / TMEM gather-decode (sm_103a): the production instantiations of
// the kernel in decode_tc.cuh, and the weight-image packing.
#include "decode_tc.cuh"

namespace ntc {

size_t tc_image_bytes(uint32_t H) {
  const size_t KH = H + 16;
  return (size_t)H * kTcKA * 2 + (size_t)H * KH * 2 + (size_t)16 * KH * 2;
}

// One CTA per decoder: fp32 weights -> the shared-memory image of the tcgen05
// kernel (bias folded in as column `in` of each layer's B operand).
template <typename T>
__global__ void k_pack_tc(const float *w32, uint32_t H, uint32_t C, uint8_t *tc, size_t tc_stride) {
  const uint32_t d = blockIdx.x;
  const size_t P = (size_t)H * 17 + (size_t)H * (H + 1) + (size_t)C * (H + 1);
  const float *p = w32 + (size_t)d * P;
  const float *W1 = p, *b1 = W1 + H * 16, *W2 = b1 + H, *b2 = W2 + (size_t)H * H, *W3 = b2 + H,
              *b3 = W3 + (size_t)C * H;
  const uint32_t KH = H + 16;
  uint8_t *img = tc + (size_t)d * tc_stride;
  uint8_t *i1 = img, *i2 = i1 + (size_t)H * kTcKA * 2, *i3 = i2 + (size_t)H * KH * 2;
  auto put = [](uint8_t *base, uint32_t r, uint32_t k, uint32_t K, float v) {
    T h = T(v);
    *reinterpret_cast<T *>(base + core_off(r, k, K)) = h;
  };
  for (uint32_t i = threadIdx.x; i < H * kTcKA; i += blockDim.x) {
    uint32_t r = i / kTcKA, k = i % kTcKA;
    put(i1, r, k, kTcKA, k < 16 ? W1[r * 16 + k] : (k == 16 ? b1[r] : 0.0f));
  }
  for (uint32_t i = threadIdx.x; i < H * KH; i += blockDim.x) {
    uint32_t r = i / KH, k = i % KH;
    put(i2, r, k, KH, k < H ? W2[(size_t)r * H + k] : (k == H ? b2[r] : 0.0f));
  }
  for (uint32_t i = threadIdx.x; i < 16 * KH; i += blockDim.x) {
    uint32_t r = i / KH, k = i % KH;
    float v = 0.0f;
    if (r < C) v = k < H ? W3[(size_t)r * H + k] : (k == H ? b3[r] : 0.0f);
    put(i3, r, k, KH, v);
  }
}

cudaError_t launch_pack_tc(const float *w32, uint32_t D, uint32_t H, uint32_t C, bool bf16,
                           uint8_t *tc, size_t tc_stride, cudaStream_t st) {
  if (bf16) k_pack_tc<__nv_bfloat16><<<D, 256, 0, st>>>(w32, H, C, tc, tc_stride);
  else k_pack_tc<__half><<<D, 256, 0, st>>>(w32, H, C, tc, tc_stride);
  return cudaGetLastError();
}

cudaError_t launch_decode_tc(const Assets &A, const WeightImages &W, const Buckets &B, size_t n,
                             void *out, unsigned long long *err, unsigned int *status, bool bf16,
                             int num_sms, cudaStream_t st, int *launches) {
  *launches += 1;
  return dispatch_tm<false>(A, W, B, n, out, err, status, bf16, num_sms, st, nullptr);
}

}  // namespace ntc
