// Decoders of a general shape (Sec. 4's decoder and the A x B sizes of its
// MLP ablation): num_levels x channels latent features (4- or 8-channel
// grids) concatenated with a positional encoding of F frequencies, 1..4 hidden
// layers of width 16..128, ReLU or LeakyReLU, sigmoid output.
//
//   k_decode_gen_tc   bucketed 128-query tiles on tcgen05, warp-specialised:
//                     a producer warpgroup gathers each row's fp16/bf16
//                     feature row into a tensor-memory ring stage; a consumer
//                     warpgroup issues each layer's MMAs (B = the decoder's
//                     weights, staged in shared memory by one bulk copy
//                     whenever the decoder changes) and runs the epilogues:
//                     fp32 bias, activation, the next layer's A operand back
//                     into tensor memory, sigmoid and the scattered store.
//                     The producer gathers the next tiles while the consumer
//                     runs a tile's MMA chain; several CTAs per SM overlap.
//   k_decode_gen_fma  per-lane fp32 FMAs, one query per thread (the fp32
//                     precision's bucketed path, and every precision's
//                     divergent-FMA mode): the same rounding rules as the
//                     standard per-lane kernel.
#include <math.h>

#include "tcgen05.cuh"

namespace ntc {
namespace {

// act: 0 ReLU, 1 LeakyReLU, 2 LeakyReLU with 0 <= slope <= 1, where
// max(h, slope * h) is the same function: evaluated on the packed fp16/bf16
// pair (slope2 = the slope in both halves), two instructions per pair
template <bool BF16>
__device__ __forceinline__ uint32_t pack_act(float lo, float hi, uint32_t act, float slope, uint32_t slope2) {
  if (act == 2) {
    const uint32_t h = pack<BF16>(lo, hi);
    uint32_t r;
    if (BF16)
      asm("{\n.reg .b32 t;\nmul.rn.bf16x2 t, %1, %2;\nmax.bf16x2 %0, %1, t;\n}" : "=r"(r) : "r"(h), "r"(slope2));
    else
      asm("{\n.reg .b32 t;\nmul.rn.f16x2 t, %1, %2;\nmax.f16x2 %0, %1, t;\n}" : "=r"(r) : "r"(h), "r"(slope2));
    return r;
  }
  if (act == 1) {
    lo = lo > 0.0f ? lo : slope * lo;
    hi = hi > 0.0f ? hi : slope * hi;
    return pack<BF16>(lo, hi);
  }
  return pack_relu<BF16>(__float_as_uint(lo), __float_as_uint(hi));
}

// LeakyReLU (0 <= slope <= 1) of the fp16 pair h + b: max(t, slope * t)
__device__ __forceinline__ uint32_t act_h2(uint32_t h, uint32_t b, uint32_t slope2) {
  uint32_t r;
  asm("{\n.reg .b32 t, u;\nadd.rn.f16x2 t, %1, %2;\nmul.rn.f16x2 u, t, %3;\nmax.f16x2 %0, t, u;\n}"
      : "=r"(r)
      : "r"(h), "r"(b), "r"(slope2));
  return r;
}

__device__ __forceinline__ void count_bad_warp(bool bad, unsigned long long *err) {
  const unsigned m = __ballot_sync(0xFFFFFFFFu, bad);
  if (m && (threadIdx.x & 31) == __ffs(m) - 1) atomicAdd(err, (unsigned long long)__popc(m));
}

// byte offset of hidden layer l's weights (l >= 1) and of the output layer's
__device__ __forceinline__ uint32_t gen_w_off(const GenWeights &G, uint32_t l) {
  return G.hidden * G.k1 * 2 + (l - 1) * G.hidden * G.hidden * 2;
}

// Dynamic shared memory: the decoder image, then (when they fit) copies of the
// tile table and of the grid table, then the ring's output rows.
constexpr uint32_t kGenTileTable = 1024;  // D + 2 entries
constexpr uint32_t kGenGrids = 1024;      // sets x levels x mips entries
constexpr uint32_t kGenStages = 2;        // tiles between the producer and the consumer
inline __host__ __device__ size_t gen_tables_off(uint32_t img_bytes) { return ((size_t)img_bytes + 15) / 16 * 16; }
inline __host__ __device__ size_t gen_oidx_off(uint32_t img_bytes) {
  return gen_tables_off(img_bytes) + 2 * kGenTileTable * 4 + (size_t)kGenGrids * sizeof(GridDesc);
}
// two output-row slots per stage (by use parity): the producer's next use of a
// stage writes the other slot, so no consumer warp reads a later tile's rows
inline __host__ __device__ size_t gen_smem_bytes(uint32_t img_bytes) {
  return gen_oidx_off(img_bytes) + (size_t)kGenStages * 2 * 128 * 4;
}

// Tensor memory: the accumulator (H columns), the hidden layers' A operand
// (H / 2 columns) and the ring's layer-1 A operands (K1 / 2 columns each).
__host__ __device__ inline uint32_t gen_tmem_need(uint32_t H, uint32_t K1) {
  return H + H / 2 + kGenStages * (K1 / 2);
}

// Warp-specialised: warpgroup 0 produces, warpgroup 1 consumes.  The CTA's
// tiles are a contiguous range t_j = t0 + j of the tile list (the latents of
// these decoders are small enough to stay in L2, so there is no locality to
// gain from neighbouring CTAs sharing tiles; consecutive tiles share their
// decoder instead); tile j goes through ring stage
// j mod kGenStages.  Producer thread r gathers row r of tile j into the stage's
// A operand (TMEM lane r) and its output row into oidx; each producer warp
// arrives on full[s].  The consumer's thread 0 issues layer 1 from the stage
// (its completion empties the stage) and every further layer from the hidden
// operand; consumer thread r runs row r's epilogues.
template <bool BF16, int L, int C>
__global__ void __launch_bounds__(256, L * C <= 4 ? 4 : (L * C <= 8 ? 3 : 2)) k_decode_gen_tc(Assets A, GenWeights G, Buckets B, void *out,
                                                       unsigned long long *err, unsigned int *status,
                                                       uint32_t tmem_cols, uint32_t img_bytes) {
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ uint64_t bars[2 * kGenStages + 2];  // full[S], empty[S], MMA completion, weight copy
  __shared__ uint32_t tmem_slot;
  __shared__ volatile uint32_t abort_flag;
  __shared__ volatile uint32_t stop_flag[2];  // the consumer's decision for tile j, in slot j & 1
  const uint32_t tid = threadIdx.x, row = tid & 127, wg = tid >> 7;
  const uint32_t lanes = ((row >> 5) * 32) << 16;  // this warp's TMEM lane quadrant
  constexpr int NF = L * C + 4 * kGenMaxPe;  // feature values this input layout can have
  constexpr int NP = (NF + 15) / 16 * 16;
  const uint32_t D = A.num_decoders, H = G.hidden, K1 = G.k1, NL = G.layers;
  const uint32_t OC = G.out_dim;
  const float *bias = reinterpret_cast<const float *>(smem + (size_t)gen_w_off(G, NL) + 16u * H * 2u);
  uint8_t *tables = smem + gen_tables_off(img_bytes);
  uint32_t *oidx = reinterpret_cast<uint32_t *>(smem + gen_oidx_off(img_bytes));
  auto full_bar = [&](uint32_t s) { return saddr(&bars[s]); };
  auto empty_bar = [&](uint32_t s) { return saddr(&bars[kGenStages + s]); };
  const uint32_t mma_bar = saddr(&bars[2 * kGenStages]), w_bar = saddr(&bars[2 * kGenStages + 1]);
  if (tid == 0) {
    for (uint32_t i = 0; i < kGenStages; ++i) {
      mbar_init(full_bar(i), 4);   // one arrival per producer warp
      mbar_init(empty_bar(i), 1);  // the layer-1 commit (or the consumer, for a tile of bad rows)
    }
    mbar_init(mma_bar, 1);
    mbar_init(w_bar, 1);
    abort_flag = 0;
    stop_flag[0] = stop_flag[1] = 0;
    asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
  }
  if (tid < 32) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(saddr(&tmem_slot)),
                 "r"(tmem_cols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
  }
  // tile and grid tables in shared memory when they fit
  const uint32_t *seg = B.meta + 1, *tst = B.meta + 1 + (D + 2);
  if (D + 2 <= kGenTileTable) {
    uint32_t *s_seg = reinterpret_cast<uint32_t *>(tables), *s_tst = s_seg + kGenTileTable;
    for (uint32_t i = tid; i < D + 2; i += blockDim.x) {
      s_seg[i] = __ldg(seg + i);
      s_tst[i] = __ldg(tst + i);
    }
    seg = s_seg;
    tst = s_tst;
  }
  const GridDesc *grids = A.grids;
  const uint32_t ngrids = A.num_sets * A.num_levels * A.num_mips;
  if (ngrids <= kGenGrids) {
    GridDesc *s_grids = reinterpret_cast<GridDesc *>(tables + 2 * kGenTileTable * 4);
    for (uint32_t i = tid; i < ngrids; i += blockDim.x) s_grids[i] = A.grids[i];
    grids = s_grids;
  }
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tAcc = tmem_slot;             // H fp32 columns
  const uint32_t tAH = tmem_slot + H;          // hidden A operand, H / 2 columns
  const uint32_t tA1 = tmem_slot + H + H / 2;  // ring stages, K1 / 2 columns each
  const uint32_t T = __ldg(B.meta);
  const bool copied = rows_copied(B, D);
  const uint32_t grid = gridDim.x;
  // this CTA's tiles: a contiguous range t0 .. t0 + K - 1 of the tile list, so
  // consecutive tiles share their decoder and the weights are copied rarely
  const uint32_t per = T / grid, rem = T % grid;
  const uint32_t t0 = blockIdx.x * per + min(blockIdx.x, rem);
  const uint32_t K = per + (blockIdx.x < rem ? 1u : 0u);
  if (wg == 0) {
    // ------------------------------------------------------------- producer
    TileWalk walk;
    // this thread's row of tile jj: its output row (kNoRow past the tile's
    // end) and query record; the bad bucket (set id out of range) is rejected
    // by query_bad().  The next tile's are loaded while tile j is gathered.
    constexpr uint32_t kNoRow = 0xFFFFFFFFu;  // never a row: n <= 2^32 - 256
    auto fetch_row = [&](uint32_t jj, uint32_t &oi_, ntc_query &q_) {
      oi_ = kNoRow;
      if (jj >= K) return;
      uint32_t d_, st_, len_;
      walk.at(seg, tst, D, t0 + jj, d_, st_, len_);
      if (row < len_) bucket_row(B, copied, st_ + row, oi_, q_);
    };
    uint32_t oi;
    ntc_query q;
    fetch_row(0, oi, q);
    for (uint32_t j = 0; j < K; ++j) {
      if (abort_flag) break;
      const uint32_t s = j % kGenStages, use = j / kGenStages;
      uint32_t noi;
      ntc_query nq;
      fetch_row(j + 1, noi, nq);
      const bool valid = oi != kNoRow;
      const bool good = valid && !query_bad(A, q);
      const bool bad = valid && !good;
      count_bad_warp(bad, err);
      if (bad) put_nan_row(out, oi, OC, G.out_half);
      // the feature row, packed to fp16/bf16 pairs as it is produced: the
      // latent features, then sin/cos pairs of the encoding (zeros beyond)
      constexpr int LW = L * C / 2, NW = NP / 2;
      uint32_t pk[NW];
#pragma unroll
      for (int i = 0; i < NW; ++i) pk[i] = 0u;
      if (good) {
        {
          __half2 hl[LW];
          gen_latents_h2<L, C>(A, grids, q, hl);
#pragma unroll
          for (int i = 0; i < LW; ++i) {
            if (BF16) {
              const float2 x = __half22float2(hl[i]);
              pk[i] = pack<true>(x.x, x.y);
            } else {
              pk[i] = *reinterpret_cast<const uint32_t *>(&hl[i]);
            }
          }
        }
        const uint32_t F = A.pe_frequencies;
        if (F) {
          // sin/cos(2 pi u) from the hardware approximation, after reducing u
          // to [-1/2, 1/2] (exact), where its absolute error is about 2^-21:
          // far below the fp16/bf16 rounding the features then go through
          float u, v, su, cu, sv, cv;
          pe_coords(A, q, u, v);
          __sincosf(6.28318530718f * __fsub_rn(u, rintf(u)), &su, &cu);
          __sincosf(6.28318530718f * __fsub_rn(v, rintf(v)), &sv, &cv);
#pragma unroll
          for (int k = 0; k < kGenMaxPe; ++k) {
            if (LW + 2 * k + 1 >= NW) break;
            if (k < (int)F) {
              pk[LW + 2 * k] = pack<BF16>(su, cu);
              pk[LW + 2 * k + 1] = pack<BF16>(sv, cv);
              const float su2 = 2.0f * su * cu, cu2 = cu * cu - su * su;
              const float sv2 = 2.0f * sv * cv, cv2 = cv * cv - sv * sv;
              su = su2, cu = cu2, sv = sv2, cv = cv2;
            }
          }
        }
      }
      if (!mbar_wait(empty_bar(s), (use & 1u) ^ 1u)) {  // the stage's previous tile has left layer 1
        atomicOr(status, 1u);
        abort_flag = 1;
      }
      fence_after();
      // (a tile of the bad bucket is stored too: its rows are zeros and the
      // consumer multiplies nothing)
#pragma unroll
      for (int kc = 0; kc < NP / 16; ++kc) {
        if ((uint32_t)kc * 16 >= K1) break;
        uint32_t p[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) p[i] = pk[8 * kc + i];
        tmem_st8(tA1 + s * (K1 / 2) + lanes + 8 * kc, p);
      }
      tmem_wait_st();
      oidx[(s * 2 + (use & 1u)) * 128 + row] = good ? oi : 0xFFFFFFFFu;
      fence_before();
      __syncwarp();
      if ((row & 31) == 0) mbar_arrive(full_bar(s));
      q = nq;
      oi = noi;
    }
  } else {
    // ------------------------------------------------------------- consumer
    uint32_t cur = 0xFFFFFFFFu, mph = 0, wph = 0;
    const uint32_t sW = saddr(smem);
    TileWalk cwalk;
    const uint32_t id_h = instr_desc<BF16>(H), id_o = instr_desc<BF16>(16);
    const uint32_t act = G.activation == 1 && G.slope >= 0.0f && G.slope <= 1.0f ? 2u : G.activation;
    const uint32_t slope2 = pack<BF16>(G.slope, G.slope);
    auto wait = [&](uint32_t bar, uint32_t parity) {
      if (!mbar_wait(bar, parity)) {
        atomicOr(status, 1u);
        abort_flag = 1;
      }
    };
    // the MMA chain: one warp waits (suspended in the barrier wait, so it
    // takes no issue slots from the producer), the named barrier releases the
    // rest of the warpgroup
    auto wait_mma = [&]() {
      if (row < 32 && !mbar_wait(mma_bar, mph)) {
        atomicOr(status, 1u);
        abort_flag = 1;
      }
      mph ^= 1;
      wg_bar(1);
    };
    for (uint32_t j = 0; j < K; ++j) {
      const uint32_t s = j % kGenStages, use = j / kGenStages;
      uint32_t dec, st, len;
      cwalk.at(seg, tst, D, t0 + j, dec, st, len);
      if (row < 32) wait(full_bar(s), use & 1u);
      // one decision to stop per tile, the same for every warp of the warpgroup
      if (row == 0) stop_flag[j & 1] = abort_flag;
      wg_bar(1);
      fence_after();
      if (stop_flag[j & 1]) break;
      const uint32_t oi = oidx[(s * 2 + (use & 1u)) * 128 + row];
      const bool good = oi != 0xFFFFFFFFu;
      if (dec >= D) {  // a tile of bad rows: nothing to multiply
        if (row == 0) mbar_arrive(empty_bar(s));
        continue;
      }
      if (dec != cur) {
        // every MMA of the previous tile has completed: the weights may change
        if (row == 0) {
          asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(w_bar), "r"(img_bytes)
                       : "memory");
          asm volatile(
              "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];\n" ::"r"(sW),
              "l"(G.tc + (size_t)dec * G.tc_stride), "r"(img_bytes), "r"(w_bar)
              : "memory");
        }
        wait(w_bar, wph);
        wph ^= 1;
        cur = dec;
      }
      if (row == 0) {
        fence_after();
        const uint64_t d1 = smem_desc(sW, K1);
        for (uint32_t kc = 0; kc < K1 / 16; ++kc)
          umma_ta(tAcc, tA1 + s * (K1 / 2) + 8 * kc, d1 + 16 * kc, id_h, kc);
        umma_commit(mma_bar);
        umma_commit(empty_bar(s));
      }
      for (uint32_t l = 0; l < NL; ++l) {
        // hidden layer l is in the accumulator: bias, activation, next A operand
        wait_mma();
        fence_after();
        const float4 *bl = reinterpret_cast<const float4 *>(bias + l * H);  // 16-byte aligned
        // fp16 with LeakyReLU: bias and activation on the packed pair
        const uint4 *bh = reinterpret_cast<const uint4 *>(bias + NL * H + 16) + l * H / 8;
        if (!BF16 && act == 2) {
          for (uint32_t c0 = 0; c0 < H; c0 += 16) {
            uint32_t v[16];
            tmem_ld16(tAcc + lanes + c0, v);
            tmem_wait_ld();
            uint32_t p[8];
#pragma unroll
            for (int i = 0; i < 2; ++i) {
              const uint4 b = bh[c0 / 8 + i];
              p[4 * i] = act_h2(pack<false>(__uint_as_float(v[8 * i]), __uint_as_float(v[8 * i + 1])), b.x, slope2);
              p[4 * i + 1] =
                  act_h2(pack<false>(__uint_as_float(v[8 * i + 2]), __uint_as_float(v[8 * i + 3])), b.y, slope2);
              p[4 * i + 2] =
                  act_h2(pack<false>(__uint_as_float(v[8 * i + 4]), __uint_as_float(v[8 * i + 5])), b.z, slope2);
              p[4 * i + 3] =
                  act_h2(pack<false>(__uint_as_float(v[8 * i + 6]), __uint_as_float(v[8 * i + 7])), b.w, slope2);
            }
            tmem_st8(tAH + lanes + c0 / 2, p);
          }
        } else if (H == 16) {
          uint32_t v[16];
          tmem_ld16(tAcc + lanes, v);
          tmem_wait_ld();
          uint32_t p[8];
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const float4 b = bl[i];
            p[2 * i] = pack_act<BF16>(__uint_as_float(v[4 * i]) + b.x, __uint_as_float(v[4 * i + 1]) + b.y, act,
                                      G.slope, slope2);
            p[2 * i + 1] = pack_act<BF16>(__uint_as_float(v[4 * i + 2]) + b.z, __uint_as_float(v[4 * i + 3]) + b.w,
                                          act, G.slope, slope2);
          }
          tmem_st8(tAH + lanes, p);
        } else {
          for (uint32_t c0 = 0; c0 < H; c0 += 32) {
            uint32_t v[32];
            tmem_ld32(tAcc + lanes + c0, v);
            tmem_wait_ld();
            uint32_t p[16];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              const float4 b = bl[c0 / 4 + i];
              p[2 * i] = pack_act<BF16>(__uint_as_float(v[4 * i]) + b.x, __uint_as_float(v[4 * i + 1]) + b.y, act,
                                        G.slope, slope2);
              p[2 * i + 1] = pack_act<BF16>(__uint_as_float(v[4 * i + 2]) + b.z, __uint_as_float(v[4 * i + 3]) + b.w,
                                            act, G.slope, slope2);
            }
            tmem_st16(tAH + lanes + c0 / 2, p);
          }
        }
        tmem_wait_st();
        fence_before();
        wg_bar(1);
        if (row == 0) {
          fence_after();
          const bool last = l + 1 == NL;
          const uint64_t dw = smem_desc(sW + gen_w_off(G, l + 1), H);
          for (uint32_t kc = 0; kc < H / 16; ++kc)
            umma_ta(tAcc, tAH + 8 * kc, dw + 16 * kc, last ? id_o : id_h, kc);
          umma_commit(mma_bar);
        }
      }
      wait_mma();
      fence_after();
      uint32_t o[16];
      tmem_ld16(tAcc + lanes, o);
      tmem_wait_ld();
      if (good) {
        const float4 *bo = reinterpret_cast<const float4 *>(bias + NL * H);
#pragma unroll
        for (int c = 0; c < 16; ++c) {
          if (c < (int)OC) {
            // sigmoid(x) = 0.5 + 0.5 * tanh(x / 2)
            const float4 b = bo[c / 4];
            const float x = __uint_as_float(o[c]) + (c % 4 == 0 ? b.x : c % 4 == 1 ? b.y : c % 4 == 2 ? b.z : b.w);
            float th;
            asm("tanh.approx.f32 %0, %1;" : "=f"(th) : "f"(0.5f * x));
            put_out(out, (size_t)oi * OC + c, fmaf(0.5f, th, 0.5f), G.out_half);
          }
        }
      }
      // the next tile's barrier (after its stage is full) orders these reads of
      // the accumulator before its layer 1 overwrites it
      fence_before();
    }
  }
  fence_before();
  __syncthreads();
  if (tid < 32) {
    fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(tmem_slot), "r"(tmem_cols)
                 : "memory");
  }
}

template <typename T>
struct Op;
template <>
struct Op<float> {
  static __device__ __forceinline__ float ld(const float *p) { return __ldg(p); }
  static __device__ __forceinline__ float round(float x) { return x; }
  static __device__ __forceinline__ float cvt(float x) { return x; }
};
template <>
struct Op<__half> {
  static __device__ __forceinline__ float ld(const __half *p) { return __half2float(__ldg(p)); }
  static __device__ __forceinline__ float round(float x) { return __half2float(__float2half_rn(x)); }
  static __device__ __forceinline__ __half cvt(float x) { return __float2half_rn(x); }
};
template <>
struct Op<__nv_bfloat16> {
  static __device__ __forceinline__ float ld(const __nv_bfloat16 *p) { return __bfloat162float(__ldg(p)); }
  static __device__ __forceinline__ float round(float x) { return __bfloat162float(__float2bfloat16_rn(x)); }
  static __device__ __forceinline__ __nv_bfloat16 cvt(float x) { return __float2bfloat16_rn(x); }
};

__device__ __forceinline__ float act_f(float x, uint32_t act, float slope) {
  return x > 0.0f ? x : (act == 1 ? slope * x : 0.0f);
}

// Per-lane decode of a general shape; row i is row i of the bucketed order B
// (bucketed != 0) or query i of qs itself, written to its output row.
template <typename T>
__global__ void __launch_bounds__(128) k_decode_gen_fma(Assets A, GenWeights G, const ntc_query *qs, int bucketed,
                                                        Buckets B, size_t n, float *out, unsigned long long *err) {
  const bool copied = bucketed && rows_copied(B, A.num_decoders);
  using E = Op<T>;
  const uint32_t H = G.hidden, I = G.in_dim, C = G.out_dim, NL = G.layers, CP = out_pad(C);
  const size_t wbytes = (((size_t)H * I + (size_t)(NL - 1) * H * H + (size_t)H * CP) * sizeof(T) + 15) / 16 * 16;
  const size_t step = (size_t)gridDim.x * blockDim.x;
  const size_t nr = (n + 31) & ~(size_t)31;  // whole warps iterate together
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < nr; i += step) {
    const bool valid = i < n;
    ntc_query q;
    uint32_t oi = 0;
    bool bad = false;
    if (valid) {
      if (bucketed) {
        bucket_row(B, copied, (uint32_t)i, oi, q);
      } else {
        q = load_query(qs + i);
        oi = (uint32_t)i;
      }
      bad = query_bad(A, q);
    }
    count_bad_warp(valid && bad, err);
    if (!valid) continue;
    float *o_row = out + (size_t)oi * C;
    if (bad) {
      for (uint32_t c = 0; c < C; ++c) o_row[c] = __int_as_float(0x7fc00000);
      continue;
    }
    const uint8_t *img = G.fma + (size_t)__ldg(A.map + q.set_id) * G.fma_stride;
    const T *W = reinterpret_cast<const T *>(img);
    const float *bias = reinterpret_cast<const float *>(img + wbytes);
    float f[kGenMaxIn];
    gen_features(A, A.grids, q, f);
    float h[kGenMaxHidden], g[kGenMaxHidden];
    for (uint32_t j = 0; j < H; ++j) {
      float acc = 0.0f;
      for (uint32_t k = 0; k < I; ++k) acc = fmaf(E::ld(W + (size_t)j * I + k), E::round(f[k]), acc);
      h[j] = E::round(act_f(acc + __ldg(bias + j), G.activation, G.slope));
    }
    const T *Wl = W + (size_t)H * I;
    for (uint32_t l = 1; l < NL; ++l) {
      for (uint32_t j = 0; j < H; ++j) {
        float acc = 0.0f;
        for (uint32_t k = 0; k < H; ++k) acc = fmaf(E::ld(Wl + (size_t)j * H + k), h[k], acc);
        g[j] = E::round(act_f(acc + __ldg(bias + l * H + j), G.activation, G.slope));
      }
      for (uint32_t j = 0; j < H; ++j) h[j] = g[j];
      Wl += (size_t)H * H;
    }
    const T *Wo = Wl;  // W_out^T [H][CP]
    for (uint32_t c = 0; c < C; ++c) {
      float acc = 0.0f;
      for (uint32_t j = 0; j < H; ++j) acc = fmaf(E::ld(Wo + (size_t)j * CP + c), h[j], acc);
      o_row[c] = 1.0f / (1.0f + expf(-(acc + __ldg(bias + NL * H + c))));
    }
  }
}

// One CTA per decoder: fp32 weights (W1, b1, {W_l, b_l}..., Wout, bout) ->
// the tcgen05 image (if tc) and the per-lane image of type T.
template <typename T>
__global__ void k_pack_gen(const float *w32, GenWeights G, uint8_t *tc, uint8_t *fma) {
  using E = Op<T>;
  const uint32_t d = blockIdx.x, H = G.hidden, I = G.in_dim, C = G.out_dim, NL = G.layers, K1 = G.k1;
  const uint32_t CP = out_pad(C);
  const size_t P = (size_t)H * I + H + (size_t)(NL - 1) * (H * H + H) + (size_t)C * H + C;
  const float *p = w32 + (size_t)d * P;
  // source offsets of each layer
  auto Wsrc = [&](uint32_t l) -> const float * {  // l = 0: W1; 1..NL-1: hidden; NL: output
    return l == 0 ? p : p + (size_t)H * I + H + (size_t)(l - 1) * (H * H + H);
  };
  auto bsrc = [&](uint32_t l) -> const float * {
    return l == 0 ? p + (size_t)H * I : Wsrc(l) + (size_t)(l < NL ? H : C) * H;
  };
  if (tc) {
    uint8_t *img = tc + (size_t)d * G.tc_stride;
    // W1 [H][K1]
    for (uint32_t e = threadIdx.x; e < H * K1; e += blockDim.x) {
      const uint32_t r = e / K1, k = e % K1;
      const float x = k < I ? Wsrc(0)[(size_t)r * I + k] : 0.0f;
      *reinterpret_cast<T *>(img + core_off(r, k, K1)) = E::cvt(x);
    }
    for (uint32_t l = 1; l <= NL; ++l) {
      const uint32_t rows = l < NL ? H : 16;
      uint8_t *base = img + (size_t)H * K1 * 2 + (size_t)(l - 1) * H * H * 2;
      for (uint32_t e = threadIdx.x; e < rows * H; e += blockDim.x) {
        const uint32_t r = e / H, k = e % H;
        const float x = (l < NL || r < C) ? Wsrc(l)[(size_t)r * H + k] : 0.0f;
        *reinterpret_cast<T *>(base + core_off(r, k, H)) = E::cvt(x);
      }
    }
    float *b = reinterpret_cast<float *>(img + gen_tc_weight_bytes(I, H, NL));
    for (uint32_t e = threadIdx.x; e < NL * H + 16; e += blockDim.x) {
      const uint32_t l = e / H;
      b[e] = l < NL ? bsrc(l)[e % H] : (e - NL * H < C ? bsrc(NL)[e - NL * H] : 0.0f);
    }
    __half *bh = reinterpret_cast<__half *>(b + NL * H + 16);
    for (uint32_t e = threadIdx.x; e < NL * H; e += blockDim.x) bh[e] = __float2half_rn(bsrc(e / H)[e % H]);
  }
  T *o = reinterpret_cast<T *>(fma + (size_t)d * G.fma_stride);
  for (uint32_t e = threadIdx.x; e < H * I; e += blockDim.x) o[e] = E::cvt(Wsrc(0)[e]);
  T *ol = o + (size_t)H * I;
  for (uint32_t l = 1; l < NL; ++l, ol += (size_t)H * H)
    for (uint32_t e = threadIdx.x; e < H * H; e += blockDim.x) ol[e] = E::cvt(Wsrc(l)[e]);
  for (uint32_t e = threadIdx.x; e < H * CP; e += blockDim.x) {
    const uint32_t j = e / CP, c = e % CP;
    ol[e] = E::cvt(c < C ? Wsrc(NL)[(size_t)c * H + j] : 0.0f);
  }
  const size_t wbytes = (((size_t)H * I + (size_t)(NL - 1) * H * H + (size_t)H * CP) * sizeof(T) + 15) / 16 * 16;
  float *ob = reinterpret_cast<float *>(fma + (size_t)d * G.fma_stride + wbytes);
  for (uint32_t e = threadIdx.x; e < NL * H + CP; e += blockDim.x) {
    const uint32_t l = e / H;
    ob[e] = l < NL ? bsrc(l)[e % H] : (e - NL * H < C ? bsrc(NL)[e - NL * H] : 0.0f);
  }
}

uint32_t gen_tmem_cols(const GenWeights &G) {
  const uint32_t need = gen_tmem_need(G.hidden, G.k1);
  uint32_t c = 32;
  while (c < need) c <<= 1;
  return c;
}

template <bool BF16, int L, int C>
cudaError_t launch_gen_tc_t(const Assets &A, const GenWeights &G, const Buckets &B, size_t n, void *out,
                            unsigned long long *err, unsigned int *status, int num_sms, cudaStream_t st) {
  const uint32_t img = (uint32_t)gen_tc_image_bytes(G.in_dim, G.hidden, G.layers);
  const size_t smem = gen_smem_bytes(img);
  const uint32_t cols = gen_tmem_cols(G);
  cudaError_t e =
      cudaFuncSetAttribute(k_decode_gen_tc<BF16, L, C>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  // resident CTAs per SM: registers, shared memory, threads, and tensor memory
  // (every resident CTA allocates `cols` of the SM's 512 columns)
  int occ = resident_ctas(k_decode_gen_tc<BF16, L, C>, 256, smem);
  occ = min(occ, (int)(512 / cols));
  if (occ < 1) occ = 1;
  const size_t max_tiles = (n + kTile - 1) / kTile + A.num_decoders + 1;
  size_t grid = (size_t)num_sms * occ;
  if (grid > max_tiles) grid = max_tiles;
  k_decode_gen_tc<BF16, L, C><<<(unsigned)grid, 256, smem, st>>>(A, G, B, out, err, status, cols, img);
  return cudaGetLastError();
}

template <bool BF16>
cudaError_t launch_gen_tc_b(const Assets &A, const GenWeights &G, const Buckets &B, size_t n, void *out,
                            unsigned long long *err, unsigned int *status, int num_sms, cudaStream_t st) {
  if (A.channels == 8)
    return A.num_levels == 2 ? launch_gen_tc_t<BF16, 2, 8>(A, G, B, n, out, err, status, num_sms, st)
                             : launch_gen_tc_t<BF16, 1, 8>(A, G, B, n, out, err, status, num_sms, st);
  return A.num_levels == 2 ? launch_gen_tc_t<BF16, 2, 4>(A, G, B, n, out, err, status, num_sms, st)
                           : launch_gen_tc_t<BF16, 1, 4>(A, G, B, n, out, err, status, num_sms, st);
}

template <typename T>
cudaError_t launch_gen_fma_t(const Assets &A, const GenWeights &G, const Buckets *B, const ntc_query *q, size_t n,
                             float *out, unsigned long long *err, int num_sms, cudaStream_t st) {
  int occ = 1;
  occ = resident_ctas(k_decode_gen_fma<T>, 128, 0);
  if (occ < 1) occ = 1;
  const size_t blocks = (n + 127) / 128;
  size_t grid = (size_t)num_sms * occ * 4;
  if (grid > blocks) grid = blocks;
  k_decode_gen_fma<T><<<(unsigned)grid, 128, 0, st>>>(A, G, q, B ? 1 : 0, B ? *B : Buckets{}, n, out, err);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_decode_gen_tc(const Assets &A, const GenWeights &G, const Buckets &B, size_t n, void *out,
                                 unsigned long long *err, unsigned int *status, bool bf16, int num_sms,
                                 cudaStream_t st, int *launches) {
  *launches += 1;
  return bf16 ? launch_gen_tc_b<true>(A, G, B, n, out, err, status, num_sms, st)
              : launch_gen_tc_b<false>(A, G, B, n, out, err, status, num_sms, st);
}

cudaError_t launch_decode_gen_fma(const Assets &A, const GenWeights &G, const Buckets *B, const ntc_query *q,
                                  size_t n, float *out, unsigned long long *err, ntc_precision prec, int num_sms,
                                  cudaStream_t st, int *launches) {
  *launches += 1;
  if (prec == NTC_PREC_FP32) return launch_gen_fma_t<float>(A, G, B, q, n, out, err, num_sms, st);
  if (prec == NTC_PREC_TC_BF16) return launch_gen_fma_t<__nv_bfloat16>(A, G, B, q, n, out, err, num_sms, st);
  return launch_gen_fma_t<__half>(A, G, B, q, n, out, err, num_sms, st);
}

cudaError_t launch_pack_gen(const float *w32, uint32_t D, const GenWeights &G, ntc_precision prec, uint8_t *tc,
                            uint8_t *fma, cudaStream_t st) {
  if (prec == NTC_PREC_FP32)
    k_pack_gen<float><<<D, 256, 0, st>>>(w32, G, nullptr, fma);
  else if (prec == NTC_PREC_TC_BF16)
    k_pack_gen<__nv_bfloat16><<<D, 256, 0, st>>>(w32, G, tc, fma);
  else
    k_pack_gen<__half><<<D, 256, 0, st>>>(w32, G, tc, fma);
  return cudaGetLastError();
}

}  // namespace ntc
