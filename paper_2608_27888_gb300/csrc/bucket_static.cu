// Allocation-free bucketing entry point.
//
// Some callers cannot allocate device memory when they need a decode sorted:
// a renderer that runs the decode inside its frame loop typically hands every
// byte of GPU memory to its own allocator up front and forbids cudaMalloc (and
// cudaMallocAsync) afterwards, because an allocation there can stall the frame
// or fail half-way through it.  ntc_bucket_static gives them the stable
// counting sort by decoder id (the same kernels as ntc_decode and
// ntc_debug_bucket) without a context and without allocating: a copy of the
// set->decoder map, the tile table with the totals and the ticket, and the
// per-chunk counts and offsets live in one file-scope device array of fixed
// size that every GPU loading this library keeps until the process exits.
#include <mutex>

#include "ntc_internal.cuh"

namespace ntc {
void set_last_error(const char *msg);  // the message ntc_last_error() returns
}

using namespace ntc;

namespace {

constexpr size_t kMapWords = 65536;    // set->decoder map copy
constexpr size_t kMetaWords = 12544;   // tile table, totals, ticket, divergence sum (<= 12295 words for D <= 4095)
constexpr size_t kCountWords = 262144; // (D+1) * ceil(n / 2048) per-chunk counts, and as many offsets
constexpr size_t kStaticWords = kMapWords + kMetaWords + 2 * kCountWords;  // 2,409,472 bytes

// The scratch.  In host code this name is only a host-side stand-in: kernels
// receive the device address looked up with cudaGetSymbolAddress below.
static __device__ __align__(256) uint32_t g_bucket_scratch[kStaticWords];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
uint32_t *g_addr[kMaxDevices] = {};

ntc_status failed(ntc_status s, const char *m) {
  set_last_error(m);
  return s;
}

}  // namespace

extern "C" NTC_API ntc_status ntc_bucket_static(const uint32_t *h_set_to_decoder, uint32_t num_sets,
                                                uint32_t num_decoders, const ntc_query *d_queries,
                                                size_t n, uint32_t *d_perm, ntc_query *d_sorted,
                                                void *cuda_stream) {
  if (!h_set_to_decoder) return failed(NTC_ERR_INVALID_ARG, "null set_to_decoder");
  if (num_sets < 1 || num_sets > kMapWords)
    return failed(NTC_ERR_INVALID_ARG, "num_sets must be in 1..65536");
  if (num_decoders < 1 || num_decoders > NTC_MAX_DECODERS)
    return failed(NTC_ERR_INVALID_ARG, "num_decoders must be in 1..4095");
  if (n > 0xFFFFFF00ull) return failed(NTC_ERR_INVALID_ARG, "too many queries");
  if (n == 0) return NTC_OK;
  if (!d_queries || !d_perm || !d_sorted) return failed(NTC_ERR_INVALID_ARG, "null device pointer");
  if (((uintptr_t)d_queries & 15) || ((uintptr_t)d_sorted & 15))
    return failed(NTC_ERR_INVALID_ARG, "query buffers must be 16-byte aligned");
  if (bucket_count_words(num_decoders, n) > kCountWords)
    return failed(NTC_ERR_UNSUPPORTED,
                  "(num_decoders + 1) * ceil(n / 2048) exceeds the static scratch (262144 counts)");
  for (uint32_t s = 0; s < num_sets; ++s)
    if (h_set_to_decoder[s] >= num_decoders)
      return failed(NTC_ERR_INVALID_ARG, "set_to_decoder entry is not a decoder");

  // set-up, once per device, with that device current
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
    return failed(NTC_ERR_CUDA, "no usable current CUDA device");
  uint32_t *base = nullptr;
  {
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_addr[dev]) {
      void *p = nullptr;
      cudaError_t e = cudaGetSymbolAddress(&p, g_bucket_scratch);
      if (e != cudaSuccess) return failed(NTC_ERR_CUDA, cudaGetErrorString(e));
      g_addr[dev] = static_cast<uint32_t *>(p);
    }
    base = g_addr[dev];
  }
  cudaStream_t st = (cudaStream_t)cuda_stream;
  uint32_t *map = base;
  uint32_t *meta = base + kMapWords;
  uint32_t *counts = meta + kMetaWords;
  uint32_t *offs = counts + kCountWords;
  // the map copy, and the tile table, totals and ticket cleared (the ticket
  // must start at 0)
  cudaError_t e = cudaMemcpyAsync(map, h_set_to_decoder, (size_t)num_sets * 4, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(meta, 0, bucket_meta_words(num_decoders) * 4, st);
  if (e != cudaSuccess) return failed(NTC_ERR_CUDA, cudaGetErrorString(e));
  Assets A{};
  A.map = map;
  A.num_sets = num_sets;
  A.num_decoders = num_decoders;
  Scratch s;
  s.perm = d_perm;
  s.meta = meta;
  s.counts = counts;
  s.offs = offs;
  s.sorted = d_sorted;
  s.dec = nullptr;  // no room for a decoder per query: the placement reads the staged records
  int launches = 0;
  e = launch_bucket(A, d_queries, n, s, st, &launches, 1);  // d_sorted is always written
  if (e != cudaSuccess) return failed(NTC_ERR_CUDA, cudaGetErrorString(e));
  return NTC_OK;
}
