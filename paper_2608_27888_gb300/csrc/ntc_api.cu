// The C ABI of libntc (declared in include/ntc.h): argument validation, device
// copies of the assets, scratch management and the launch sequence of each
// decode path.
#include <stdarg.h>
#include <stdlib.h>
#include <stdio.h>
#include <string.h>

#include <vector>

#include "ntc_internal.cuh"
#include "tcgen05.cuh"

using namespace ntc;

// ntc_decode_host splits a batch into at most kHostChunks pipelined chunks of
// at least kHostChunkMin queries.
constexpr int kHostChunks = 32;
constexpr size_t kHostChunkMin = 1u << 18;

struct ntc_ctx {
  int device = 0;
  int num_sms = 0;
  uint32_t S = 0, D = 0, M = 0, H = 0, C = 0, address_mode = 0;
  // decoder shape; `general` is every shape but the standard one (2 levels x 8
  // channels, no encoding, 2 hidden layers of 64 or 128, ReLU)
  uint32_t L = kLevels, LC = kChannels, F = 0, NL = 2, in_dim = kInDim, act = 0;
  float slope = 0.0f;
  bool general = false;
  uint32_t out_half = 0;  // output rows are IEEE half (NTC_OUTPUT_FP16)
  uint8_t *d_gtc = nullptr, *d_gfma = nullptr;
  size_t gtc_stride = 0, gfma_stride = 0;
  ntc_precision prec = NTC_PREC_TC_FP16;
  uint64_t num_texels = 0;
  uint4 *d_lat = nullptr;
  GridDesc *d_grids = nullptr;
  uint4 *d_pair = nullptr;      // row-pair copy of the latents, 32 B per texel
  GridDesc *d_pgrids = nullptr;  // grid bases in d_pair
  uint32_t *d_map = nullptr;
  uint8_t *d_mma = nullptr;
  float *d_f32 = nullptr;
  uint8_t *d_tc = nullptr;
  uint8_t *d_fma = nullptr;
  size_t mma_stride = 0, f32_stride = 0, tc_stride = 0, fma_stride = 0;
  unsigned long long *d_err = nullptr;
  unsigned int *d_status = nullptr;  // nonzero: a decode kernel gave up a bounded wait
  // bucketing scratch (grows on demand, stream-ordered)
  size_t cap_n = 0, cap_counts = 0;
  uint32_t *d_perm = nullptr, *d_meta = nullptr, *d_counts = nullptr;
  ntc_query *d_sorted = nullptr;
  void *d_dec = nullptr;  // decoder per query (1 or 2 bytes)
  // staging for ntc_decode_host, and its copy streams and chunk events
  size_t cap_host = 0;
  ntc_query *d_hq = nullptr;
  uint8_t *d_hout = nullptr;  // [cap_host][C] output elements of out_bytes each
  cudaStream_t s_up = nullptr, s_down = nullptr;
  cudaEvent_t ev_begin = nullptr, ev_up = nullptr, ev_done = nullptr;
  uint64_t launches = 0;
  // optional stage timing
  bool timing = false;
  bool timed = false;
  cudaEvent_t ev[3] = {nullptr, nullptr, nullptr};
};

static thread_local char g_err[512] = "";

static ntc_status fail(ntc_status s, const char *fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof g_err, fmt, ap);
  va_end(ap);
  return s;
}

namespace ntc {
void set_last_error(const char *msg) { snprintf(g_err, sizeof g_err, "%s", msg); }
bool pdl_enabled() {
  static const bool on = getenv("NTC_NO_PDL") == nullptr;
  return on;
}
}  // namespace ntc

static ntc_status cuda_fail(cudaError_t e, const char *what) {
  if (e == cudaErrorMemoryAllocation)
    return fail(NTC_ERR_OUT_OF_MEMORY, "%s: %s", what, cudaGetErrorString(e));
  return fail(NTC_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

#define CK(call, what)                            \
  do {                                            \
    cudaError_t e_ = (call);                      \
    if (e_ != cudaSuccess) return cuda_fail(e_, what); \
  } while (0)

namespace {

// Keeps the caller's current device and restores it.
struct DeviceGuard {
  int prev = -1;
  bool ok = true;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
    if (prev != dev) ok = cudaSetDevice(dev) == cudaSuccess;
  }
  ~DeviceGuard() {
    int now = -1;
    if (prev >= 0 && cudaGetDevice(&now) == cudaSuccess && now != prev) cudaSetDevice(prev);
  }
};

Assets assets_of(const ntc_ctx *c) {
  Assets A;
  A.lat = c->d_lat;
  A.grids = c->d_grids;
  A.pair = c->d_pair;
  A.pgrids = c->d_pgrids;
  A.map = c->d_map;
  A.num_sets = c->S;
  A.num_decoders = c->D;
  A.num_mips = c->M;
  A.address_mode = c->address_mode;
  A.num_levels = c->L;
  A.channels = c->LC;
  A.pe_frequencies = c->F;
  return A;
}

GenWeights gen_of(const ntc_ctx *c) {
  GenWeights G;
  G.tc = c->d_gtc;
  G.tc_stride = c->gtc_stride;
  G.fma = c->d_gfma;
  G.fma_stride = c->gfma_stride;
  G.in_dim = c->in_dim;
  G.k1 = gen_k1(c->in_dim);
  G.hidden = c->H;
  G.layers = c->NL;
  G.out_dim = c->C;
  G.activation = c->act;
  G.slope = c->slope;
  G.out_half = c->out_half;
  return G;
}

WeightImages weights_of(const ntc_ctx *c) {
  WeightImages W;
  W.mma = c->d_mma;
  W.mma_stride = c->mma_stride;
  W.f32 = c->d_f32;
  W.f32_stride = c->f32_stride;
  W.tc = c->d_tc;
  W.tc_stride = c->tc_stride;
  W.fma = c->d_fma;
  W.fma_stride = c->fma_stride;
  W.hidden = c->H;
  W.out_dim = c->C;
  W.out_half = c->out_half;
  return W;
}

void release(ntc_ctx *c) {
  for (auto &e : c->ev)
    if (e) cudaEventDestroy(e);
  if (c->ev_up) cudaEventDestroy(c->ev_up);
  if (c->ev_done) cudaEventDestroy(c->ev_done);
  if (c->ev_begin) cudaEventDestroy(c->ev_begin);
  if (c->s_up) cudaStreamDestroy(c->s_up);
  if (c->s_down) cudaStreamDestroy(c->s_down);
  cudaFree(c->d_lat);
  cudaFree(c->d_grids);
  cudaFree(c->d_pair);
  cudaFree(c->d_pgrids);
  cudaFree(c->d_map);
  cudaFree(c->d_mma);
  cudaFree(c->d_f32);
  cudaFree(c->d_tc);
  cudaFree(c->d_fma);
  cudaFree(c->d_gtc);
  cudaFree(c->d_gfma);
  cudaFree(c->d_err);
  cudaFree(c->d_status);
  cudaFree(c->d_perm);
  cudaFree(c->d_meta);
  cudaFree(c->d_counts);
  cudaFree(c->d_sorted);
  cudaFree(c->d_dec);
  cudaFree(c->d_hq);
  cudaFree(c->d_hout);
}

size_t round16(size_t x) { return (x + 15) & ~(size_t)15; }

// Make sure the bucketing scratch holds n queries (stream-ordered
// allocation): perm, the sorted query records and the decoder ids [n], the
// per-chunk counts and offsets (one allocation, offsets in its second half),
// and the tile table with the totals, the ticket and the divergence sum
// (zeroed once; the bucketing leaves them at zero).
ntc_status ensure_scratch(ntc_ctx *c, size_t n, cudaStream_t st) {
  const size_t counts = bucket_count_words(c->D, n);
  if (!c->d_meta) {
    const size_t words = bucket_meta_words(c->D);
    CK(cudaMallocAsync((void **)&c->d_meta, words * 4, st), "scratch allocation");
    CK(cudaMemsetAsync(c->d_meta, 0, words * 4, st), "scratch clear");
  }
  if (counts > c->cap_counts) {
    if (c->d_counts) CK(cudaFreeAsync(c->d_counts, st), "scratch free");
    c->d_counts = nullptr;
    c->cap_counts = 0;
    CK(cudaMallocAsync((void **)&c->d_counts, 2 * counts * 4, st), "scratch allocation");
    c->cap_counts = counts;
  }
  if (n > c->cap_n) {
    if (c->d_perm) CK(cudaFreeAsync(c->d_perm, st), "scratch free");
    if (c->d_sorted) CK(cudaFreeAsync(c->d_sorted, st), "scratch free");
    if (c->d_dec) CK(cudaFreeAsync(c->d_dec, st), "scratch free");
    c->d_perm = nullptr;
    c->d_sorted = nullptr;
    c->d_dec = nullptr;
    c->cap_n = 0;
    CK(cudaMallocAsync((void **)&c->d_perm, n * 4, st), "scratch allocation");
    CK(cudaMallocAsync((void **)&c->d_sorted, n * sizeof(ntc_query), st), "scratch allocation");
    CK(cudaMallocAsync(&c->d_dec, n * bucket_dec_bytes(c->D), st), "scratch allocation");
    c->cap_n = n;
  }
  return NTC_OK;
}

Scratch scratch_of(const ntc_ctx *c) {
  Scratch s;
  s.perm = c->d_perm;
  s.meta = c->d_meta;
  s.counts = c->d_counts;
  s.offs = c->d_counts + c->cap_counts;
  s.sorted = c->d_sorted;
  s.dec = c->d_dec;
  return s;
}

ntc_status check_queries(const ntc_ctx *ctx, const void *q, size_t n) {
  if (!ctx) return fail(NTC_ERR_INVALID_ARG, "null context");
  if (n > 0xFFFFFF00ull) return fail(NTC_ERR_INVALID_ARG, "n = %zu exceeds 2^32 - 256 queries", n);
  if (n && !q) return fail(NTC_ERR_INVALID_ARG, "null query pointer");
  if (((uintptr_t)q & 15) != 0) return fail(NTC_ERR_INVALID_ARG, "query buffer is not 16-byte aligned");
  return NTC_OK;
}

// The failure path of every bounded wait, run on purpose: an mbarrier whose
// phase 0 nothing completes (one expected arrival, none made), waited for with
// the kernels' own mbar_wait, which returns false once kWaitLimitNs has passed;
// the give-up sets status bit 0 as a decode kernel's would.
__global__ void k_wait_timeout(unsigned int *status) {
  __shared__ uint64_t bar;
  const uint32_t b = ntc::saddr(&bar);
  ntc::mbar_init(b, 1);
  asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
  if (!ntc::mbar_wait(b, 0)) atomicOr(status, 1u);
}

}  // namespace

extern "C" {

const char *ntc_last_error(void) { return g_err; }

const char *ntc_status_string(ntc_status s) {
  switch (s) {
    case NTC_OK: return "ok";
    case NTC_ERR_INVALID_ARG: return "invalid argument";
    case NTC_ERR_UNSUPPORTED: return "unsupported";
    case NTC_ERR_OUT_OF_MEMORY: return "out of memory";
    case NTC_ERR_CUDA: return "CUDA error";
  }
  return "unknown status";
}

ntc_status ntc_create(const ntc_desc *d, ntc_ctx **out) {
  if (!out) return fail(NTC_ERR_INVALID_ARG, "null output pointer");
  *out = nullptr;
  if (!d) return fail(NTC_ERR_INVALID_ARG, "null descriptor");
  if (!d->level_dims || !d->latent_offsets || !d->latents || !d->weights || !d->set_to_decoder)
    return fail(NTC_ERR_INVALID_ARG, "null array in descriptor");
  if (d->num_sets < 1) return fail(NTC_ERR_INVALID_ARG, "num_sets must be >= 1");
  if (d->num_decoders < 1 || d->num_decoders > NTC_MAX_DECODERS)
    return fail(NTC_ERR_INVALID_ARG, "num_decoders must be in 1..%u", NTC_MAX_DECODERS);
  if (d->latent_channels != 4 && d->latent_channels != 8)
    return fail(NTC_ERR_UNSUPPORTED, "latent_channels must be 4 or 8");
  if (d->num_levels != 1 && d->num_levels != 2) return fail(NTC_ERR_UNSUPPORTED, "num_levels must be 1 or 2");
  if (d->num_mips < 1 || d->num_mips > kMaxMips)
    return fail(NTC_ERR_INVALID_ARG, "num_mips must be in 1..%d", kMaxMips);
  if (d->pe_frequencies > (uint32_t)kGenMaxPe)
    return fail(NTC_ERR_UNSUPPORTED, "pe_frequencies must be at most %d", kGenMaxPe);
  if (d->in_dim != d->num_levels * d->latent_channels + 4 * d->pe_frequencies)
    return fail(NTC_ERR_INVALID_ARG, "in_dim must be num_levels * latent_channels + 4 * pe_frequencies");
  if (d->in_dim > (uint32_t)kGenMaxIn) return fail(NTC_ERR_UNSUPPORTED, "in_dim must be at most %d", kGenMaxIn);
  if (d->hidden != 16 && d->hidden != 32 && d->hidden != 64 && d->hidden != 128)
    return fail(NTC_ERR_UNSUPPORTED, "hidden must be 16, 32, 64 or 128");
  if (d->num_hidden_layers < 1 || d->num_hidden_layers > (uint32_t)kGenMaxLayers)
    return fail(NTC_ERR_UNSUPPORTED, "num_hidden_layers must be in 1..%d", kGenMaxLayers);
  if (d->out_dim < 1 || d->out_dim > 16) return fail(NTC_ERR_UNSUPPORTED, "out_dim must be in 1..16");
  if (d->activation > 1) return fail(NTC_ERR_INVALID_ARG, "activation must be 0 (ReLU) or 1 (LeakyReLU)");
  if (d->activation == 1 && !(d->leaky_slope - d->leaky_slope == 0.0f))
    return fail(NTC_ERR_INVALID_ARG, "leaky_slope must be finite");
  if (d->precision != NTC_PREC_TC_FP16 && d->precision != NTC_PREC_TC_BF16 && d->precision != NTC_PREC_FP32)
    return fail(NTC_ERR_INVALID_ARG, "unknown precision");
  if (d->address_mode > 1) return fail(NTC_ERR_INVALID_ARG, "address_mode must be 0 (wrap) or 1 (clamp)");
  if (d->output_format != NTC_OUTPUT_FP32 && d->output_format != NTC_OUTPUT_FP16)
    return fail(NTC_ERR_INVALID_ARG, "output_format must be NTC_OUTPUT_FP32 or NTC_OUTPUT_FP16");
  if (d->output_format == NTC_OUTPUT_FP16 && d->precision == NTC_PREC_FP32)
    return fail(NTC_ERR_UNSUPPORTED, "fp16 output rows come from the tensor-core precisions only");
  if (d->num_texels < 1) return fail(NTC_ERR_INVALID_ARG, "num_texels must be >= 1");
  const uint32_t S = d->num_sets, M = d->num_mips, L = d->num_levels;
  std::vector<GridDesc> grids((size_t)S * L * M);
  for (uint32_t s = 0; s < S; ++s)
    for (uint32_t k = 0; k < L; ++k) {
      const uint32_t W0 = d->level_dims[((size_t)s * L + k) * 2];
      const uint32_t H0 = d->level_dims[((size_t)s * L + k) * 2 + 1];
      if (W0 < 1 || H0 < 1 || W0 > (1u << 24) || H0 > (1u << 24) || (uint64_t)W0 * H0 > 0xFFFFFFFFull)
        return fail(NTC_ERR_INVALID_ARG, "set %u level %u: bad grid size %ux%u", s, k, W0, H0);
      for (uint32_t m = 0; m < M; ++m) {
        const uint32_t W = W0 >> m ? W0 >> m : 1, H = H0 >> m ? H0 >> m : 1;
        const uint64_t base = d->latent_offsets[((size_t)s * L + k) * M + m];
        if (base > d->num_texels || (uint64_t)W * H > d->num_texels - base)
          return fail(NTC_ERR_INVALID_ARG, "set %u level %u mip %u lies outside the latents", s, k, m);
        GridDesc &g = grids[((size_t)s * L + k) * M + m];
        g.base = base;
        g.W = W;
        g.H = H;
      }
    }
  for (uint32_t s = 0; s < S; ++s)
    if (d->set_to_decoder[s] >= d->num_decoders)
      return fail(NTC_ERR_INVALID_ARG, "set_to_decoder[%u] = %u is not a decoder", s, d->set_to_decoder[s]);

  ntc_ctx *c = new ntc_ctx;
  if (cudaGetDevice(&c->device) != cudaSuccess) {
    delete c;
    return fail(NTC_ERR_CUDA, "no CUDA device");
  }
  cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, c->device);
  c->S = S;
  c->D = d->num_decoders;
  c->M = M;
  c->H = d->hidden;
  c->C = d->out_dim;
  c->address_mode = d->address_mode;
  c->prec = d->precision;
  c->num_texels = d->num_texels;
  c->L = L;
  c->LC = d->latent_channels;
  c->F = d->pe_frequencies;
  c->NL = d->num_hidden_layers;
  c->in_dim = d->in_dim;
  c->act = d->activation;
  c->slope = d->activation == 1 ? d->leaky_slope : 0.0f;
  c->out_half = d->output_format == NTC_OUTPUT_FP16;
  c->general = !(c->L == kLevels && c->LC == kChannels && c->F == 0 && c->NL == 2 && c->act == 0 &&
                 (c->H == 64 || c->H == 128));
  const size_t P = (size_t)c->H * (c->in_dim + 1) + (size_t)(c->NL - 1) * c->H * (c->H + 1) +
                   (size_t)c->C * (c->H + 1);
  c->mma_stride = round16(mma_image_bytes(c->H));
  c->f32_stride = (f32_image_floats(c->H, c->C) + 3) & ~(size_t)3;
  c->tc_stride = round16(tc_image_bytes(c->H));
  c->fma_stride = round16(fma_image_bytes(c->H, c->C, c->prec == NTC_PREC_FP32 ? 4u : 2u));
  c->gtc_stride = round16(gen_tc_image_bytes(c->in_dim, c->H, c->NL));
  c->gfma_stride = round16(gen_fma_image_bytes(c->in_dim, c->H, c->NL, c->C, c->prec == NTC_PREC_FP32 ? 4u : 2u));
  // the row-pair copy (standard shape only): grids back to back, built in
  // chunks of kPairChunk texels
  std::vector<GridDesc> pgrids(c->general ? 0 : grids.size());
  std::vector<uint32_t> chunk_grid, chunk_start;
  uint64_t num_pairs = 0;
  for (size_t g = 0; g < pgrids.size(); ++g) {
    pgrids[g] = grids[g];
    pgrids[g].base = num_pairs;
    const uint64_t nt = (uint64_t)grids[g].W * grids[g].H;
    num_pairs += nt;
    for (uint64_t t = 0; t < nt; t += kPairChunk) {
      chunk_grid.push_back((uint32_t)g);
      chunk_start.push_back((uint32_t)t);
    }
  }
  uint32_t *d_chunks = nullptr;
  float *d_w32 = nullptr;
  cudaError_t e = cudaSuccess;
  auto step = [&](cudaError_t r) {
    if (e == cudaSuccess) e = r;
  };
  const size_t lat_bytes = d->num_texels * d->latent_channels * 2;
  step(cudaMalloc((void **)&c->d_lat, lat_bytes));
  step(cudaMalloc((void **)&c->d_grids, grids.size() * sizeof(GridDesc)));
  step(cudaMalloc((void **)&c->d_map, (size_t)S * 4));
  step(cudaMalloc((void **)&c->d_err, sizeof(unsigned long long)));
  step(cudaMalloc((void **)&c->d_status, sizeof(unsigned int)));
  step(cudaMalloc((void **)&d_w32, P * 4 * c->D));
  if (!c->general) {
    step(cudaMalloc((void **)&c->d_mma, c->mma_stride * c->D));
    step(cudaMalloc((void **)&c->d_f32, c->f32_stride * 4 * c->D));
    step(cudaMalloc((void **)&c->d_tc, c->tc_stride * c->D));
    step(cudaMalloc((void **)&c->d_fma, c->fma_stride * c->D));
    step(cudaMalloc((void **)&c->d_pair, num_pairs * 32));
    step(cudaMalloc((void **)&c->d_pgrids, pgrids.size() * sizeof(GridDesc)));
    step(cudaMalloc((void **)&d_chunks, chunk_grid.size() * 2 * sizeof(uint32_t)));
  } else {
    if (c->prec != NTC_PREC_FP32) step(cudaMalloc((void **)&c->d_gtc, c->gtc_stride * c->D));
    step(cudaMalloc((void **)&c->d_gfma, c->gfma_stride * c->D));
  }
  if (e == cudaSuccess) {
    step(cudaMemcpy(c->d_lat, d->latents, lat_bytes, cudaMemcpyHostToDevice));
    step(cudaMemcpy(c->d_grids, grids.data(), grids.size() * sizeof(GridDesc), cudaMemcpyHostToDevice));
    step(cudaMemcpy(c->d_map, d->set_to_decoder, (size_t)S * 4, cudaMemcpyHostToDevice));
    step(cudaMemcpy(d_w32, d->weights, P * 4 * c->D, cudaMemcpyHostToDevice));
    step(cudaMemset(c->d_err, 0, sizeof(unsigned long long)));
    step(cudaMemset(c->d_status, 0, sizeof(unsigned int)));
    if (!c->general) {
      step(cudaMemcpy(c->d_pgrids, pgrids.data(), pgrids.size() * sizeof(GridDesc), cudaMemcpyHostToDevice));
      step(cudaMemcpy(d_chunks, chunk_grid.data(), chunk_grid.size() * sizeof(uint32_t), cudaMemcpyHostToDevice));
      step(cudaMemcpy(d_chunks + chunk_grid.size(), chunk_start.data(), chunk_start.size() * sizeof(uint32_t),
                      cudaMemcpyHostToDevice));
      step(launch_build_pairs(assets_of(c), d_chunks, d_chunks + chunk_grid.size(), (uint32_t)chunk_grid.size(),
                              c->d_pair, 0));
      step(cudaMemset(c->d_tc, 0, c->tc_stride * c->D));
      step(launch_pack_weights(d_w32, c->D, c->H, c->C, c->prec == NTC_PREC_TC_BF16, c->d_mma,
                               c->mma_stride, c->d_f32, c->f32_stride, c->d_tc, c->tc_stride, 0));
      step(launch_pack_fma(d_w32, c->D, c->H, c->C, c->prec, c->d_fma, c->fma_stride, 0));
    } else {
      if (c->d_gtc) step(cudaMemset(c->d_gtc, 0, c->gtc_stride * c->D));
      step(cudaMemset(c->d_gfma, 0, c->gfma_stride * c->D));
      step(launch_pack_gen(d_w32, c->D, gen_of(c), c->prec, c->d_gtc, c->d_gfma, 0));
    }
    step(cudaDeviceSynchronize());
  }
  cudaFree(d_w32);
  cudaFree(d_chunks);
  if (e != cudaSuccess) {
    release(c);
    delete c;
    return cuda_fail(e, "ntc_create");
  }
  *out = c;
  return NTC_OK;
}

ntc_status ntc_destroy(ntc_ctx *c) {
  if (!c) return NTC_OK;
  DeviceGuard g(c->device);
  cudaDeviceSynchronize();
  release(c);
  delete c;
  return NTC_OK;
}

namespace {
ntc_status decode_impl(ntc_ctx *c, const ntc_query *q, size_t n, void *out, void *stream, ntc_mode mode,
                       ntc_debug_row *rows);
}

ntc_status ntc_decode(ntc_ctx *c, const ntc_query *q, size_t n, void *out, void *stream,
                      ntc_mode mode) {
  return decode_impl(c, q, n, out, stream, mode, nullptr);
}

ntc_status ntc_debug_decode_rows(ntc_ctx *c, const ntc_query *q, size_t n, void *out, ntc_debug_row *rows,
                                 void *stream) {
  if (!c) return fail(NTC_ERR_INVALID_ARG, "null context");
  if (c->general || c->prec == NTC_PREC_FP32)
    return fail(NTC_ERR_UNSUPPORTED, "rows are recorded by the standard-shape tensor-core decode only");
  if (n && !rows) return fail(NTC_ERR_INVALID_ARG, "null rows pointer");
  return decode_impl(c, q, n, out, stream, NTC_MODE_BUCKETED, rows);
}

}  // extern "C"

namespace {
// ntc_decode; with rows != nullptr the tensor-core kernel is the debug
// instantiation that also records every row it builds.
ntc_status decode_impl(ntc_ctx *c, const ntc_query *q, size_t n, void *vout, void *stream, ntc_mode mode,
                       ntc_debug_row *rows) {
  ntc_status s = check_queries(c, q, n);
  if (s != NTC_OK) return s;
  if (n && !vout) return fail(NTC_ERR_INVALID_ARG, "null output pointer");
  if (((uintptr_t)vout & (c->out_half ? 1 : 3)) != 0)
    return fail(NTC_ERR_INVALID_ARG, "output buffer is not aligned to its element (%d bytes)", c->out_half ? 2 : 4);
  float *out = static_cast<float *>(vout);  // the fp32 paths
  if (mode != NTC_MODE_BUCKETED && mode != NTC_MODE_DIVERGENT && mode != NTC_MODE_BUCKETED_MMA &&
      mode != NTC_MODE_DIVERGENT_FMA)
    return fail(NTC_ERR_INVALID_ARG, "unknown mode");
  const bool fp32 = c->prec == NTC_PREC_FP32;
  if (fp32 && mode != NTC_MODE_BUCKETED && mode != NTC_MODE_DIVERGENT_FMA)
    return fail(NTC_ERR_UNSUPPORTED, "the fp32 precision has only the bucketed and divergent FMA modes");
  if (c->general && mode != NTC_MODE_BUCKETED && mode != NTC_MODE_DIVERGENT_FMA)
    return fail(NTC_ERR_UNSUPPORTED, "this decoder shape has only the bucketed and divergent FMA modes");
  if (c->out_half && mode != NTC_MODE_BUCKETED)
    return fail(NTC_ERR_UNSUPPORTED, "fp16 output rows are written by the bucketed tensor-core decode only");
  if (n == 0) return NTC_OK;
  DeviceGuard g(c->device);
  if (!g.ok) return fail(NTC_ERR_CUDA, "cannot select the context's device");
  cudaStream_t st = (cudaStream_t)stream;
  const Assets A = assets_of(c);
  const WeightImages W = weights_of(c);
  const bool bf16 = c->prec == NTC_PREC_TC_BF16;
  int launches = 0;
  cudaError_t e;
  const bool unsorted = mode == NTC_MODE_DIVERGENT || mode == NTC_MODE_DIVERGENT_FMA;
  // one decoder shared by every set (the paper's shared decoder): there is no
  // divergence to remove, so the tensor-core decode takes the queries in their
  // own order and nothing is sorted
  const bool shared = mode == NTC_MODE_BUCKETED && !fp32 && !c->general && c->D == 1;
  s = unsorted || shared ? NTC_OK : ensure_scratch(c, n, st);
  if (s != NTC_OK) return s;
  if (c->timing) CK(cudaEventRecord(c->ev[0], st), "event record");
  if (unsorted) {
    if (c->timing) CK(cudaEventRecord(c->ev[1], st), "event record");
    if (c->general)
      e = launch_decode_gen_fma(A, gen_of(c), nullptr, q, n, out, c->d_err, c->prec, c->num_sms, st, &launches);
    else if (mode == NTC_MODE_DIVERGENT)
      e = launch_decode_divergent(A, W, q, n, out, c->d_err, bf16, c->num_sms, st, &launches);
    else
      e = launch_decode_divergent_fma(A, W, q, n, out, c->d_err, c->prec, c->num_sms, st, &launches);
    c->launches += launches;
    if (e != cudaSuccess) return cuda_fail(e, "divergent decode launch");
    if (c->timing) {
      CK(cudaEventRecord(c->ev[2], st), "event record");
      c->timed = true;
    }
    return NTC_OK;
  }
  Buckets B;
  if (shared) {
    B.queries = q;
    B.perm = nullptr;
    B.meta = nullptr;
    B.identity_n = (uint32_t)n;
  } else {
    e = launch_bucket(A, q, n, scratch_of(c), st, &launches);
    if (e != cudaSuccess) {
      c->launches += launches;
      return cuda_fail(e, "bucketing launch");
    }
    B.queries = q;
    B.sorted = c->d_sorted;
    B.perm = c->d_perm;
    B.meta = c->d_meta;
  }
  if (c->timing) CK(cudaEventRecord(c->ev[1], st), "event record");
  if (c->general && fp32)
    e = launch_decode_gen_fma(A, gen_of(c), &B, nullptr, n, out, c->d_err, c->prec, c->num_sms, st, &launches);
  else if (c->general)
    e = launch_decode_gen_tc(A, gen_of(c), B, n, vout, c->d_err, c->d_status, bf16, c->num_sms, st, &launches);
  else if (fp32)
    e = launch_decode_fp32(A, W, B, n, out, c->d_err, c->num_sms, st, &launches);
  else if (mode == NTC_MODE_BUCKETED_MMA)
    e = launch_decode_mma(A, W, B, n, out, c->d_err, bf16, c->num_sms, st, &launches);
  else if (rows)
    e = launch_decode_tc_debug(A, W, B, n, vout, c->d_err, c->d_status, bf16, c->num_sms, st, &launches, rows);
  else
    e = launch_decode_tc(A, W, B, n, vout, c->d_err, c->d_status, bf16, c->num_sms, st, &launches);
  c->launches += launches;
  if (e != cudaSuccess) return cuda_fail(e, "decode launch");
  if (c->timing) {
    CK(cudaEventRecord(c->ev[2], st), "event record");
    c->timed = true;
  }
  return NTC_OK;
}
}  // namespace

extern "C" {

ntc_status ntc_decode_host(ntc_ctx *c, const ntc_query *hq, size_t n, void *vhout, void *stream,
                           ntc_mode mode) {
  uint8_t *hout = static_cast<uint8_t *>(vhout);
  ntc_status s = check_queries(c, hq, n);
  if (s != NTC_OK) return s;
  if (n && !hout) return fail(NTC_ERR_INVALID_ARG, "null output pointer");
  if (n == 0) return NTC_OK;
  DeviceGuard g(c->device);
  cudaStream_t st = (cudaStream_t)stream;
  if (n > c->cap_host) {
    CK(cudaStreamSynchronize(st), "staging resize");
    if (c->s_up) CK(cudaStreamSynchronize(c->s_up), "staging resize");
    if (c->s_down) CK(cudaStreamSynchronize(c->s_down), "staging resize");
    cudaFree(c->d_hq);
    cudaFree(c->d_hout);
    c->d_hq = nullptr;
    c->d_hout = nullptr;
    c->cap_host = 0;
    CK(cudaMalloc((void **)&c->d_hq, n * sizeof(ntc_query)), "staging allocation");
    CK(cudaMalloc((void **)&c->d_hout, n * c->C * (c->out_half ? 2 : 4)), "staging allocation");
    c->cap_host = n;
  }
  if (!c->s_up) {
    CK(cudaStreamCreateWithFlags(&c->s_up, cudaStreamNonBlocking), "copy stream");
    CK(cudaStreamCreateWithFlags(&c->s_down, cudaStreamNonBlocking), "copy stream");
    CK(cudaEventCreateWithFlags(&c->ev_begin, cudaEventDisableTiming), "chunk event");
    CK(cudaEventCreateWithFlags(&c->ev_up, cudaEventDisableTiming), "chunk event");
    CK(cudaEventCreateWithFlags(&c->ev_done, cudaEventDisableTiming), "chunk event");
  }
  // Chunks pipeline the upload (s_up), the decode (the caller's stream) and the
  // download (s_down): chunk i+1 uploads and chunk i-1 downloads while chunk i
  // decodes.  Each chunk is bucketed on its own; every query's output is the
  // same as in one call over all n.  One event per direction serves every
  // chunk: a stream wait takes the event's latest record when it is enqueued.
  size_t chunk = (n + kHostChunks - 1) / kHostChunks;
  if (chunk < kHostChunkMin) chunk = kHostChunkMin;
  chunk = (chunk + kBucketChunk - 1) / kBucketChunk * kBucketChunk;
  const size_t nchunks = (n + chunk - 1) / chunk;
  const size_t row = (size_t)c->C * (c->out_half ? 2 : 4);  // bytes of one output row
  CK(cudaEventRecord(c->ev_begin, st), "chunk event");
  CK(cudaStreamWaitEvent(c->s_up, c->ev_begin, 0), "stream order");
  CK(cudaStreamWaitEvent(c->s_down, c->ev_begin, 0), "stream order");
  for (size_t i = 0; i < nchunks; ++i) {
    const size_t off = i * chunk, m = n - off < chunk ? n - off : chunk;
    CK(cudaMemcpyAsync(c->d_hq + off, hq + off, m * sizeof(ntc_query), cudaMemcpyHostToDevice, c->s_up),
       "query upload");
    CK(cudaEventRecord(c->ev_up, c->s_up), "chunk event");
    CK(cudaStreamWaitEvent(st, c->ev_up, 0), "stream order");
    s = ntc_decode(c, c->d_hq + off, m, c->d_hout + off * row, stream, mode);
    if (s != NTC_OK) {
      cudaStreamSynchronize(c->s_up);
      cudaStreamSynchronize(c->s_down);
      return s;
    }
    CK(cudaEventRecord(c->ev_done, st), "chunk event");
    CK(cudaStreamWaitEvent(c->s_down, c->ev_done, 0), "stream order");
    CK(cudaMemcpyAsync(hout + off * row, c->d_hout + off * row, m * row, cudaMemcpyDeviceToHost, c->s_down),
       "output download");
  }
  CK(cudaStreamSynchronize(c->s_down), "decode");
  CK(cudaStreamSynchronize(st), "decode");
  return NTC_OK;
}

ntc_status ntc_debug_taps(ntc_ctx *c, const ntc_query *q, size_t n, uint64_t *idx, float *w,
                          float *t, void *stream) {
  ntc_status s = check_queries(c, q, n);
  if (s != NTC_OK) return s;
  if (n && (!idx || !w || !t)) return fail(NTC_ERR_INVALID_ARG, "null output pointer");
  if (n == 0) return NTC_OK;
  DeviceGuard g(c->device);
  int launches = 0;
  cudaError_t e = launch_debug_taps(assets_of(c), q, n, (unsigned long long *)idx, w, t,
                                    (cudaStream_t)stream, &launches);
  c->launches += launches;
  if (e != cudaSuccess) return cuda_fail(e, "debug taps launch");
  return NTC_OK;
}

ntc_status ntc_debug_features(ntc_ctx *c, const ntc_query *q, size_t n, float *f, void *stream) {
  ntc_status s = check_queries(c, q, n);
  if (s != NTC_OK) return s;
  if (n && !f) return fail(NTC_ERR_INVALID_ARG, "null output pointer");
  if (n == 0) return NTC_OK;
  DeviceGuard g(c->device);
  int launches = 0;
  cudaError_t e = launch_debug_features(assets_of(c), q, n, f, (cudaStream_t)stream, &launches);
  c->launches += launches;
  if (e != cudaSuccess) return cuda_fail(e, "debug features launch");
  return NTC_OK;
}

size_t ntc_max_tiles(const ntc_ctx *c, size_t n) {
  if (!c) return 0;
  return (n + kTile - 1) / kTile + c->D + 1;
}

ntc_status ntc_debug_bucket(ntc_ctx *c, const ntc_query *q, size_t n, uint32_t *perm,
                            uint32_t *counts, uint32_t *tiles, uint32_t *num_tiles, uint32_t *divergence,
                            void *stream) {
  ntc_status s = check_queries(c, q, n);
  if (s != NTC_OK) return s;
  if (n && !perm) return fail(NTC_ERR_INVALID_ARG, "null perm pointer");
  DeviceGuard g(c->device);
  cudaStream_t st = (cudaStream_t)stream;
  int launches = 0;
  if (n == 0) {
    if (counts) CK(cudaMemsetAsync(counts, 0, (c->D + 1) * 4, st), "clear");
    if (num_tiles) CK(cudaMemsetAsync(num_tiles, 0, 4, st), "clear");
    if (divergence) CK(cudaMemsetAsync(divergence, 0, 8, st), "clear");
    return NTC_OK;
  }
  s = ensure_scratch(c, n, st);
  if (s != NTC_OK) return s;
  cudaError_t e = launch_bucket(assets_of(c), q, n, scratch_of(c), st, &launches);
  if (e == cudaSuccess) e = cudaMemcpyAsync(perm, c->d_perm, n * 4, cudaMemcpyDeviceToDevice, st);
  if (e == cudaSuccess && (counts || tiles || num_tiles))
    e = launch_tiles_export(c->d_meta, c->D, tiles, num_tiles, counts, ntc_max_tiles(c, n), st, &launches);
  if (e == cudaSuccess && divergence)  // the words copied, divergence are adjacent
    e = cudaMemcpyAsync(divergence, c->d_meta + meta_copied(c->D), 8, cudaMemcpyDeviceToDevice, st);
  c->launches += launches;
  if (e != cudaSuccess) return cuda_fail(e, "bucketing");
  return NTC_OK;
}

ntc_status ntc_get_error_count(ntc_ctx *c, uint64_t *count) {
  if (!c || !count) return fail(NTC_ERR_INVALID_ARG, "null argument");
  DeviceGuard g(c->device);
  CK(cudaDeviceSynchronize(), "synchronize");
  unsigned long long v = 0;
  unsigned int st = 0;
  CK(cudaMemcpy(&v, c->d_err, sizeof v, cudaMemcpyDeviceToHost), "error counter read");
  CK(cudaMemcpy(&st, c->d_status, sizeof st, cudaMemcpyDeviceToHost), "status read");
  *count = v;
  if (st) return fail(NTC_ERR_CUDA, "a decode kernel gave up waiting for the tensor core; results are invalid");
  return NTC_OK;
}

ntc_status ntc_reset_error_count(ntc_ctx *c) {
  if (!c) return fail(NTC_ERR_INVALID_ARG, "null context");
  DeviceGuard g(c->device);
  CK(cudaDeviceSynchronize(), "synchronize");
  CK(cudaMemset(c->d_err, 0, sizeof(unsigned long long)), "error counter reset");
  CK(cudaMemset(c->d_status, 0, sizeof(unsigned int)), "status reset");
  return NTC_OK;
}

ntc_status ntc_debug_wait_timeout(ntc_ctx *c, void *stream) {
  if (!c) return fail(NTC_ERR_INVALID_ARG, "null context");
  DeviceGuard g(c->device);
  k_wait_timeout<<<1, 1, 0, (cudaStream_t)stream>>>(c->d_status);
  c->launches += 1;
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "wait-timeout launch");
  return NTC_OK;
}

uint64_t ntc_launch_count(const ntc_ctx *c) { return c ? c->launches : 0; }

ntc_status ntc_set_stage_timing(ntc_ctx *c, int enable) {
  if (!c) return fail(NTC_ERR_INVALID_ARG, "null context");
  DeviceGuard g(c->device);
  if (enable && !c->ev[0])
    for (auto &e : c->ev) CK(cudaEventCreate(&e), "event create");
  c->timing = enable != 0;
  c->timed = false;
  return NTC_OK;
}

ntc_status ntc_stage_times(ntc_ctx *c, float times[2]) {
  if (!c || !times) return fail(NTC_ERR_INVALID_ARG, "null argument");
  if (!c->timed) return fail(NTC_ERR_INVALID_ARG, "no timed decode since timing was enabled");
  DeviceGuard g(c->device);
  CK(cudaEventSynchronize(c->ev[2]), "event synchronize");
  CK(cudaEventElapsedTime(&times[0], c->ev[0], c->ev[1]), "event elapsed");
  CK(cudaEventElapsedTime(&times[1], c->ev[1], c->ev[2]), "event elapsed");
  return NTC_OK;
}

}  // extern "C"
