// tcgen05 / TMEM gather-decode (sm_103a).
//
// One persistent CTA per SM holds NWG warpgroups; each warpgroup decodes its own
// single-decoder 128-query tiles (tiles are dealt out round-robin over all
// warpgroups of the grid, so at any moment the whole GPU works on neighbouring
// tiles -- the same decoder and, for a set-major bucket order, the same
// latents, which keeps them in L2).  Per tile:
//   1. each thread gathers its query's latent taps, blends them in fp32 and
//      writes one fp16/bf16 row of the A tile [128 x 32] (16 features, a 1 in
//      column 16 that multiplies the bias row of the weights, zeros) into
//      shared memory;
//   2. one thread issues the layer-1 tcgen05.mma (M=128, N=H, K=32) into the
//      warpgroup's TMEM columns and commits to an mbarrier;
//   3. the four warps read their 32 TMEM lanes (tcgen05.ld), apply ReLU while
//      converting to fp16/bf16, and write the hidden tile [128 x (H+16)] (with
//      its own ones column) to shared memory; layer 2 (N=H) and layer 3 (N=16)
//      follow the same way; the last epilogue applies the sigmoid and scatters
//      the rows to out[perm[i]].
// Shared-memory operands use the no-swizzle K-major canonical layout: 8-row x
// 16-byte core matrices, K-adjacent core matrices 128 B apart (LBO), 8-row
// groups K*16 B apart (SBO).  The decoder's weights (bias folded in as an extra
// K column) are copied from a pre-packed image whenever a warpgroup's tile
// changes decoder.  Every mbarrier wait is bounded by time; on expiry the
// kernel records an error and stops cleanly (TMEM is always released).
#include "ntc_internal.cuh"

namespace ntc {

constexpr int kTcKA = 32;  // K of the A tile: 16 features + bias column + pad
constexpr uint64_t kWaitLimitNs = 200ull * 1000ull * 1000ull;

size_t tc_image_bytes(uint32_t H) {
  const size_t KH = H + 16;
  return (size_t)H * kTcKA * 2 + (size_t)H * KH * 2 + (size_t)16 * KH * 2;
}

// byte offset of element (r, k) in a no-swizzle K-major tile with K columns
__host__ __device__ __forceinline__ uint32_t core_off(uint32_t r, uint32_t k, uint32_t K) {
  return (r >> 3) * (K * 16) + (k >> 3) * 128 + (r & 7) * 16 + (k & 7) * 2;
}

namespace {

__device__ __forceinline__ uint32_t saddr(const void *p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n.reg .pred p;\nmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      "selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Wait for the phase with the given parity to complete; false after the limit.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  while (!mbar_try_wait(bar, parity))
    if (global_ns() - t0 > kWaitLimitNs) return false;
  return true;
}

__device__ __forceinline__ void fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
}
__device__ __forceinline__ void fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
}
__device__ __forceinline__ void fence_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
}
__device__ __forceinline__ void wg_bar(int wg) {
  asm volatile("bar.sync %0, 128;\n" ::"r"(wg + 1) : "memory");
}

__device__ __forceinline__ uint64_t smem_desc(uint32_t addr, uint32_t K) {
  return (uint64_t)((addr >> 4) & 0x3FFFu) | ((uint64_t)(128u >> 4) << 16) |
         ((uint64_t)(((K * 16u) >> 4) & 0x3FFFu) << 32) | (1ull << 46);
}

template <bool BF16>
__host__ __device__ constexpr uint32_t instr_desc(uint32_t N) {
  return (1u << 4) | ((BF16 ? 1u : 0u) << 7) | ((BF16 ? 1u : 0u) << 10) | ((N >> 3) << 17) |
         ((128u >> 4) << 24);
}

__device__ __forceinline__ void umma(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                     uint32_t accum) {
  asm volatile(
      "{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(a), "l"(b), "r"(idesc), "r"(accum)
      : "memory");
}

__device__ __forceinline__ void umma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(bar)
               : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]),
        "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]),
        "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15},"
      " [%16];\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}

__device__ __forceinline__ void tmem_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
}

template <bool BF16>
__device__ __forceinline__ uint32_t pack_relu(uint32_t lo, uint32_t hi) {
  uint32_t r;
  if (BF16) asm("cvt.rn.relu.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(__uint_as_float(hi)), "f"(__uint_as_float(lo)));
  else asm("cvt.rn.relu.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(__uint_as_float(hi)), "f"(__uint_as_float(lo)));
  return r;
}

template <bool BF16>
__device__ __forceinline__ uint32_t pack(float lo, float hi) {
  uint32_t r;
  if (BF16) asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  else asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

__device__ __forceinline__ void sts128(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};\n" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d)
               : "memory");
}

// TMEM accumulator row (H fp32 columns) -> ReLU -> fp16/bf16 hidden tile row.
template <int H, bool BF16>
__device__ __forceinline__ void epilogue_hidden(uint32_t tmem_row, uint32_t sH, uint32_t row) {
  constexpr uint32_t KH = H + 16;
#pragma unroll
  for (int c0 = 0; c0 < H; c0 += 64) {
    uint32_t a[32], b[32];
    tmem_ld32(tmem_row + c0, a);
    tmem_ld32(tmem_row + c0 + 32, b);
    tmem_wait_ld();
#pragma unroll
    for (int i = 0; i < 4; ++i)
      sts128(sH + core_off(row, c0 + 8 * i, KH), pack_relu<BF16>(a[8 * i], a[8 * i + 1]),
             pack_relu<BF16>(a[8 * i + 2], a[8 * i + 3]), pack_relu<BF16>(a[8 * i + 4], a[8 * i + 5]),
             pack_relu<BF16>(a[8 * i + 6], a[8 * i + 7]));
#pragma unroll
    for (int i = 0; i < 4; ++i)
      sts128(sH + core_off(row, c0 + 32 + 8 * i, KH), pack_relu<BF16>(b[8 * i], b[8 * i + 1]),
             pack_relu<BF16>(b[8 * i + 2], b[8 * i + 3]), pack_relu<BF16>(b[8 * i + 4], b[8 * i + 5]),
             pack_relu<BF16>(b[8 * i + 6], b[8 * i + 7]));
  }
}

template <int H>
struct TcLayout {
  static constexpr uint32_t KH = H + 16;
  static constexpr uint32_t W1 = H * kTcKA * 2;
  static constexpr uint32_t W2 = H * KH * 2;
  static constexpr uint32_t W3 = 16 * KH * 2;
  static constexpr uint32_t WIMG = W1 + W2 + W3;
  static constexpr uint32_t A = 128 * kTcKA * 2;
  static constexpr uint32_t HT = 128 * KH * 2;
  static constexpr uint32_t WG = WIMG + A + HT;  // shared bytes per warpgroup
};

template <int H, int NWG, bool BF16>
__global__ void __launch_bounds__(NWG * 128, 1)
    k_decode_tc(Assets A, WeightImages W, Buckets B, float *out, unsigned long long *err,
                unsigned int *status) {
  using L = TcLayout<H>;
  extern __shared__ __align__(128) uint8_t smem[];
  const int wg = threadIdx.x >> 7, tid = threadIdx.x & 127, warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  uint8_t *my = smem + (size_t)wg * L::WG;
  const uint32_t sW1 = saddr(my), sW2 = sW1 + L::W1, sW3 = sW2 + L::W2, sA = sW3 + L::W3,
                 sH = sA + L::A;
  uint64_t *bars = reinterpret_cast<uint64_t *>(smem + (size_t)NWG * L::WG);
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bars + NWG);
  volatile uint32_t *abort_flag = tmem_slot + 1;  // [NWG]
  constexpr uint32_t kCols = NWG * H;             // 256
  const uint32_t bar = saddr(bars + wg);

  if (threadIdx.x == 0) {
    for (int w = 0; w < NWG; ++w) mbar_init(saddr(bars + w), 1);
    asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
  }
  if (tid == 0) abort_flag[wg] = 0;
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(
                     saddr(tmem_slot)),
                 "r"(kCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
  }
  // constant columns: A[r][16] = 1 (bias), A[r][17..31] = 0; H[r][H] = 1, H[r][H+1..] = 0
  const uint32_t one = BF16 ? 0x3F80u : 0x3C00u;
  sts128(sA + core_off(tid, 16, kTcKA), one, 0, 0, 0);
  sts128(sA + core_off(tid, 24, kTcKA), 0, 0, 0, 0);
  sts128(sH + core_off(tid, H, L::KH), one, 0, 0, 0);
  sts128(sH + core_off(tid, H + 8, L::KH), 0, 0, 0, 0);
  fence_async_smem();
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const uint32_t tmem_wg = tmem_base + (uint32_t)(wg * H);
  const uint32_t tmem_row = tmem_wg + ((uint32_t)((warp & 3) * 32) << 16);

  const uint32_t D = A.num_decoders, C = W.out_dim;
  const uint32_t T = __ldg(B.meta);
  const uint32_t G = gridDim.x * NWG;
  uint32_t phase = 0, cur = 0xFFFFFFFFu;
  constexpr uint32_t id_hidden = instr_desc<BF16>(H), id_out = instr_desc<BF16>(16);

  for (uint32_t t = blockIdx.x * NWG + wg; t < T; t += G) {
    uint32_t dec, start, len;
    tile_info(B.meta, D, t, dec, start, len);
    const bool valid = (uint32_t)tid < len;
    ntc_query q;
    uint32_t oi = 0;
    bool bad = true;
    if (valid) {
      q = load_query(B.sorted + start + tid);
      oi = __ldg(B.perm + start + tid);
      bad = dec == D || query_bad(A, q);
    }
    const uint32_t badm = __ballot_sync(0xFFFFFFFFu, valid && bad);
    if (badm && lane == __ffs(badm) - 1) atomicAdd(err, (unsigned long long)__popc(badm));
    if (valid && bad)
      for (uint32_t c = 0; c < C; ++c) out[(size_t)oi * C + c] = __int_as_float(0x7fc00000);
    if (dec == D) continue;  // the whole tile is bad queries (uniform)

    if (dec != cur) {  // this warpgroup's previous MMAs are complete: reload weights
      const uint4 *src = reinterpret_cast<const uint4 *>(W.tc + (size_t)dec * W.tc_stride);
      uint4 *dst = reinterpret_cast<uint4 *>(my);
      for (uint32_t i = tid; i < L::WIMG / 16; i += 128) dst[i] = __ldg(src + i);
      cur = dec;
    }
    float f[kInDim];
#pragma unroll
    for (int c = 0; c < kInDim; ++c) f[c] = 0.0f;
    if (valid && !bad) query_features(A, q, f);
    sts128(sA + core_off(tid, 0, kTcKA), pack<BF16>(f[0], f[1]), pack<BF16>(f[2], f[3]),
           pack<BF16>(f[4], f[5]), pack<BF16>(f[6], f[7]));
    sts128(sA + core_off(tid, 8, kTcKA), pack<BF16>(f[8], f[9]), pack<BF16>(f[10], f[11]),
           pack<BF16>(f[12], f[13]), pack<BF16>(f[14], f[15]));
    fence_async_smem();
    wg_bar(wg);
    // layer 1: [128 x 32] x [32 x H]
    if (tid == 0) {
      fence_after();
#pragma unroll
      for (uint32_t k = 0; k < kTcKA / 16; ++k)
        umma(tmem_wg, smem_desc(sA + k * 256, kTcKA), smem_desc(sW1 + k * 256, kTcKA), id_hidden, k);
      umma_commit(bar);
    }
    if (!mbar_wait(bar, phase)) {
      atomicOr(status, 1u);
      abort_flag[wg] = 1;
    }
    phase ^= 1;
    fence_after();
    epilogue_hidden<H, BF16>(tmem_row, sH, tid);
    fence_async_smem();
    fence_before();
    wg_bar(wg);
    // layer 2: [128 x (H+16)] x [(H+16) x H]
    if (tid == 0) {
      fence_after();
#pragma unroll
      for (uint32_t k = 0; k < L::KH / 16; ++k)
        umma(tmem_wg, smem_desc(sH + k * 256, L::KH), smem_desc(sW2 + k * 256, L::KH), id_hidden, k);
      umma_commit(bar);
    }
    if (!mbar_wait(bar, phase)) {
      atomicOr(status, 1u);
      abort_flag[wg] = 1;
    }
    phase ^= 1;
    fence_after();
    epilogue_hidden<H, BF16>(tmem_row, sH, tid);
    fence_async_smem();
    fence_before();
    wg_bar(wg);
    // layer 3: [128 x (H+16)] x [(H+16) x 16]
    if (tid == 0) {
      fence_after();
#pragma unroll
      for (uint32_t k = 0; k < L::KH / 16; ++k)
        umma(tmem_wg, smem_desc(sH + k * 256, L::KH), smem_desc(sW3 + k * 256, L::KH), id_out, k);
      umma_commit(bar);
    }
    if (!mbar_wait(bar, phase)) {
      atomicOr(status, 1u);
      abort_flag[wg] = 1;
    }
    phase ^= 1;
    fence_after();
    uint32_t o[16];
    tmem_ld16(tmem_row, o);
    tmem_wait_ld();
    if (valid && !bad) {
      float *dst = out + (size_t)oi * C;
#pragma unroll
      for (int c = 0; c < 16; ++c)
        if (c < (int)C) dst[c] = 1.0f / (1.0f + __expf(-__uint_as_float(o[c])));
    }
    fence_before();
    wg_bar(wg);
    if (abort_flag[wg]) break;
  }
  fence_before();
  __syncthreads();
  if (warp == 0) {
    fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(tmem_base), "r"(kCols)
                 : "memory");
  }
}

template <int H, int NWG, bool BF16>
cudaError_t launch_tc_t(const Assets &A, const WeightImages &W, const Buckets &B, size_t n,
                        float *out, unsigned long long *err, unsigned int *status, int num_sms,
                        cudaStream_t st) {
  using L = TcLayout<H>;
  const size_t smem = (size_t)NWG * L::WG + NWG * 8 + 8 + 4 * NWG;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k_decode_tc<H, NWG, BF16>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  const size_t max_tiles = (n + kTile - 1) / kTile + A.num_decoders + 1;
  size_t grid = (size_t)num_sms;
  const size_t need = (max_tiles + NWG - 1) / NWG;
  if (grid > need) grid = need;
  k_decode_tc<H, NWG, BF16><<<(unsigned)grid, NWG * 128, smem, st>>>(A, W, B, out, err, status);
  return cudaGetLastError();
}

}  // namespace

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
                             float *out, unsigned long long *err, unsigned int *status, bool bf16,
                             int num_sms, cudaStream_t st, int *launches) {
  *launches += 1;
  if (W.hidden == 64)
    return bf16 ? launch_tc_t<64, 4, true>(A, W, B, n, out, err, status, num_sms, st)
                : launch_tc_t<64, 4, false>(A, W, B, n, out, err, status, num_sms, st);
  return bf16 ? launch_tc_t<128, 2, true>(A, W, B, n, out, err, status, num_sms, st)
              : launch_tc_t<128, 2, false>(A, W, B, n, out, err, status, num_sms, st);
}

}  // namespace ntc
