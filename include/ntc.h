/*
 * ntc.h -- C ABI of libntc, the GB300 (sm_103a) runtime decoder for
 * neural-compressed textures with shared decoders.
 *
 * Problem (Sec. 2 and Sec. 3.3 of "Thread-Efficient Decoding for Neural
 * Texture Compression"): every pixel of a rendering pass asks for a texel of
 * some texture set i; the texel is x^_i = D_{c(i)}(z_i), the latents z_i of
 * that set decoded by the MLP decoder D_g of the set's group g = c(i) (one
 * decoder per set in the non-shared baseline, one per cluster, or one shared by
 * all sets).  When one warp holds queries of several decoders it diverges
 * (Sec. 2); libntc removes that divergence by bucketing the queries by decoder
 * before the tensor-core decode, and keeps an unsorted "divergent" decode as
 * the comparison the paper measures (Sec. 4.4, Tables 5-6).
 *
 * Reading of the decode (the paper leaves the sampling rule open):
 *   - the MLP input is the concatenation of bilinear fetches from
 *     `num_levels` latent grids (Sec. 1: "latent pyramids or grids"), each an
 *     8-channel fp16 grid with its own box-filtered mip chain;
 *   - texel-centre convention x = u*W - 0.5; address_mode 0 wraps u to [0,1)
 *     and indices modulo W, 1 clamps indices to [0, W-1];
 *   - mip: lambda = max(lod, 0), lo = min(floor(lambda), num_mips-1),
 *     t = lambda - lo unless lo is the last mip (then t = 0); with t > 0 the
 *     level feature is (1-t) f(lo) + t f(lo+1) (one MLP evaluation);
 *   - address and weight arithmetic is fp32 round-to-nearest without
 *     contraction, so texel indices and bilinear weights are reproducible
 *     bit for bit;
 *   - decoder: 3-layer MLP (Sec. 4: first two layers hidden), ReLU on the
 *     hidden layers, sigmoid on the output, fp32 out.
 *
 * Memory: the context owns device copies of latents, weights and map.  Query
 * and output buffers of ntc_decode are DEVICE pointers owned by the caller.
 * Scratch (the permutation and a decoder id per query, 5 or 6 bytes per
 * query, 8 bytes per decoder and 2048 queries of chunk counts and offsets, and
 * the tile table) is owned by the context and grows on demand with cudaMallocAsync on
 * the call's stream.  Every bucketed decode sorts with the same stable
 * counting sort that ntc_debug_bucket exports.  One context must not run two
 * decodes concurrently (on different streams or threads).
 *
 * Errors: host-detectable problems return a status and enqueue nothing; the
 * message is available from ntc_last_error().  A query whose set id is out of
 * range or whose u or v is not finite decodes to NaN in every channel and is
 * counted (ntc_get_error_count).  No kernel traps.
 *
 * Environment: the bucketing kernels and the tensor-core decode after them
 * are launched as programmatic dependents of their predecessor on the stream
 * (each starts while the one before is finishing and waits for its results).
 * With NTC_NO_PDL set (any value, read once per process) they are ordinary
 * launches instead; the results are the same.  Profilers that replay a single
 * kernel of such a chain need it.
 */
#ifndef NTC_H
#define NTC_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define NTC_API __attribute__((visibility("default")))
#else
#define NTC_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef struct ntc_ctx ntc_ctx;

typedef enum {
  NTC_OK = 0,
  NTC_ERR_INVALID_ARG = 1,   /* null pointer, inconsistent sizes, bad map entry */
  NTC_ERR_UNSUPPORTED = 2,   /* a shape or mode this build does not implement  */
  NTC_ERR_OUT_OF_MEMORY = 3, /* a device allocation failed                     */
  NTC_ERR_CUDA = 4           /* any other CUDA runtime error                   */
} ntc_status;

/* One decode query, 16 bytes, in device memory: texture-set id, UV, lod. */
typedef struct {
  uint32_t set_id;
  float u, v;
  float lod;
} ntc_query;

/* Arithmetic of the MLP.  TC_*: tensor cores with fp16/bf16 operands and fp32
 * accumulation; FP32: CUDA-core fp32 reference mode.  Bias and sigmoid are
 * fp32 in every mode; the output rows are fp32 unless ntc_desc.output_format
 * asks for fp16 rows. */
typedef enum {
  NTC_PREC_TC_FP16 = 0,
  NTC_PREC_TC_BF16 = 1,
  NTC_PREC_FP32 = 2
} ntc_precision;

/* Which decode path ntc_decode runs.
 * BUCKETED:     the queries are sorted stably by decoder id (the permutation
 *               ntc_debug_bucket returns), then the gather-decode runs over
 *               128-query single-decoder tiles: the tcgen05/TMEM kernel for
 *               the tensor-core precisions, FFMA for FP32.  With one decoder
 *               for all sets the tensor-core decode takes the queries in their
 *               own order.  Each output row depends only on its own query, so
 *               the grouping never changes an output.
 * DIVERGENT:    no sorting: each warp takes 32 consecutive queries and loops over
 *               its distinct decoders (the non-shared setting of Sec. 4.4).
 *               Tensor-core precisions only.
 * BUCKETED_MMA: the bucketed path with the warp-level mma.sync decode kernel.
 *               Tensor-core precisions only.
 * DIVERGENT_FMA: no sorting and no tensor cores: every thread evaluates its
 *               own query's decoder with fp32 fused multiply-adds, weights read
 *               per lane (the "Non-Shared FMA" setting of Sec. 4.4, Tables
 *               5-6).  Every precision: with TC_FP16/TC_BF16 the features,
 *               weights and hidden activations are rounded to that type and
 *               accumulated in fp32; FP32 rounds nothing. */
typedef enum {
  NTC_MODE_BUCKETED = 0,
  NTC_MODE_DIVERGENT = 1,
  NTC_MODE_BUCKETED_MMA = 2,
  NTC_MODE_DIVERGENT_FMA = 3
} ntc_mode;

/* Everything ntc_create needs.  All pointers are HOST memory owned by the
 * caller; ntc_create copies them and keeps no reference. */
typedef struct {
  uint32_t num_sets;          /* texture sets, >= 1                            */
  uint32_t num_decoders;      /* decoders (groups), 1 .. NTC_MAX_DECODERS       */
  uint32_t latent_channels;   /* channels per latent texel: 8, or 4 (Sec. 4's
                                 256x256x4 grid)                                */
  uint32_t num_levels;        /* latent grids per set: 2, or 1                  */
  uint32_t num_mips;          /* mip-chain length of every grid, 1 .. 16        */
  const uint32_t *level_dims; /* [num_sets][num_levels][2]: W, H of mip 0       */
  const uint64_t *latent_offsets; /* [num_sets][num_levels][num_mips]: first
                                 texel of each mip in `latents` (texel units);
                                 mip m is max(1,W>>m) x max(1,H>>m) texels,
                                 row-major, channel-last                       */
  const uint16_t *latents;    /* IEEE fp16 bits, [num_texels][latent_channels] */
  uint64_t num_texels;        /* length of `latents` in texels                  */
  uint32_t in_dim;            /* = num_levels * latent_channels +
                                 4 * pe_frequencies, at most 64                 */
  uint32_t hidden;            /* hidden width: 16, 32, 64 or 128                */
  uint32_t num_hidden_layers; /* 1 .. 4 (an MLP of num_hidden_layers + 1 layers;
                                 Sec. 4 uses 2, the ablation A x B sizes vary
                                 it)                                            */
  uint32_t out_dim;           /* output channels, 1 .. 16                       */
  const float *weights;       /* [num_decoders][P], per decoder W1[hidden][in],
                                 b1[hidden], then per further hidden layer
                                 W[hidden][hidden], b[hidden], then
                                 Wout[out][hidden], bout[out] (row-major
                                 [out][in]); P = hidden*(in+1) +
                                 (num_hidden_layers-1)*hidden*(hidden+1) +
                                 out*(hidden+1)                                 */
  const uint32_t *set_to_decoder; /* [num_sets]: c(i), each < num_decoders      */
  ntc_precision precision;
  uint32_t address_mode;      /* 0 = wrap, 1 = clamp                            */
  uint32_t pe_frequencies;    /* F, 0 .. 8: the MLP input ends with the
                                 positional encoding sin/cos(2 pi 2^k u'),
                                 sin/cos(2 pi 2^k v') for k < F (u', v' the
                                 coordinates the taps use: wrapped into [0,1)
                                 in wrap mode); Sec. 4 concatenates the encoder
                                 output with a positional encoding             */
  uint32_t activation;        /* 0 = ReLU, 1 = LeakyReLU (Sec. 4)               */
  float leaky_slope;          /* LeakyReLU slope for x <= 0 (e.g. 0.01)         */
  uint32_t output_format;     /* NTC_OUTPUT_FP32 or NTC_OUTPUT_FP16, below      */
} ntc_desc;

/* Output element type of ntc_decode.  FP32: out_dim floats per row.  FP16:
 * out_dim IEEE binary16 values per row, each the fp32 sigmoid rounded to
 * nearest even (a C = 8 row is 16 bytes, one vector store); the paper's fp16
 * kernels are fp16 end to end (Sec. 4.4, Tables 5-6).  FP16 rows are written
 * by the BUCKETED mode with the tensor-core precisions (ntc_create refuses
 * FP16 rows with NTC_PREC_FP32; ntc_decode returns NTC_ERR_UNSUPPORTED for the
 * other modes).  A bad query's row is NaN (0x7E00) in every channel. */
#define NTC_OUTPUT_FP32 0u
#define NTC_OUTPUT_FP16 1u

/* Decoder shapes.  The standard shape (2 levels x 8 channels, no encoding, 2
 * hidden layers of 64 or 128, ReLU) runs every mode on the specialised
 * kernels.  Every other shape ntc_create accepts (the paper's 4-channel grid
 * with positional encoding and LeakyReLU, the A x B ablation sizes) runs the
 * BUCKETED mode (a general tcgen05 decode over the sorted tiles for fp16/bf16,
 * per-lane fp32 for FP32) and the DIVERGENT_FMA mode; the other modes return
 * NTC_ERR_UNSUPPORTED. */

#define NTC_MAX_DECODERS 4095u
#define NTC_TILE_ROWS 128u

/* Validate `desc`, copy latents, weights and map to the current CUDA device
 * and return a context in *out: the per-set latents z_{g,i}, the group
 * decoders D_g and the map c(i) of Sec. 3.3 (with Sec. 4's decoder shapes).
 * Synchronous.  On failure *out is NULL. */
NTC_API ntc_status ntc_create(const ntc_desc *desc, ntc_ctx **out);

/* Decode n queries: every query's latent features go through the MLP decoder
 * of its texture set's group -- the per-pixel decode whose divergence Sec. 2
 * measures, with the decoder D_g shared by the sets i of group g = c(i)
 * (Sec. 3.1, Sec. 3.3): d_out[i][c] = channel c of D_{c(set_i)}(features of
 * query i), for c < out_dim, in the queries' original order.
 * d_queries: device array of n records (16-byte aligned).  d_out: device
 * array of n*out_dim elements of the context's output format (floats, 4-byte
 * aligned; or IEEE halves, 2-byte aligned).  Asynchronous on `cuda_stream` (a
 * cudaStream_t; NULL is the legacy default stream); no host synchronisation.
 * n = 0 is a no-op.  Output for a bad query is NaN in every channel. */
NTC_API ntc_status ntc_decode(ntc_ctx *ctx, const ntc_query *d_queries, size_t n, void *d_out,
                      void *cuda_stream, ntc_mode mode);

/* ntc_decode on HOST buffers: copies the queries to context-owned device
 * memory, decodes, copies the outputs back into h_out and synchronises before
 * returning.  The batch is split into up to 32 chunks (at least 2^18 queries
 * each) whose upload, decode and download overlap: uploads and downloads run
 * on two context-owned streams ordered after the work already queued on
 * `cuda_stream`, decodes on `cuda_stream`.  Each chunk is bucketed on its own;
 * outputs are the same as one ntc_decode over all n.  Pinned host memory is
 * needed for the copies to overlap. */
NTC_API ntc_status ntc_decode_host(ntc_ctx *ctx, const ntc_query *h_queries, size_t n, void *h_out,
                           void *cuda_stream, ntc_mode mode);

/* Free the context and everything it owns (no paper counterpart).  NULL is
 * accepted. */
NTC_API ntc_status ntc_destroy(ntc_ctx *ctx);

/* --------------------------------------------------------------- debug / test */

/* Taps of every query by the reference addressing (the sampling of Sec. 1's
 * latent grids as the fp32, mma.sync and divergent paths compute it; the
 * default tensor-core kernel's own taps, recorded by ntc_debug_decode_rows,
 * have the same texel indices bit for bit and these weights times the mip
 * blend factor).  d_idx: [n][num_levels][2][4]
 * uint64 texel indices into `latents`; d_w: same shape, fp32 bilinear weights;
 * d_t: [n] fp32 mip blend factor.  Slot [k][0] holds mip lo, slot [k][1] mip
 * lo+1 and is filled only when t > 0 (otherwise index UINT64_MAX, weight 0);
 * a bad query reports UINT64_MAX / 0 everywhere.  Device pointers; async. */
NTC_API ntc_status ntc_debug_taps(ntc_ctx *ctx, const ntc_query *d_queries, size_t n, uint64_t *d_idx,
                          float *d_w, float *d_t, void *cuda_stream);

/* The fp32 MLP input of every query, d_feat[n][in_dim]: the latent features
 * of every level, then the positional encoding they are concatenated with
 * (Sec. 4) (NaN rows for bad queries).  Computed in fp32 from the taps above
 * (the tensor-core kernels blend in packed fp16 instead; see ntc_debug_row).
 * Device pointers; async. */
NTC_API ntc_status ntc_debug_features(ntc_ctx *ctx, const ntc_query *d_queries, size_t n, float *d_feat,
                              void *cuda_stream);

/* The bucketing stage alone (Sec. 2: the queries of one block that need
 * different decoders are what diverges; sorting by decoder leaves tiles of one
 * decoder), by the same kernels and the same scratch as ntc_decode's BUCKETED
 * mode.  d_perm[n]: query indices in (decoder, original index) order, where a
 * query with an out-of-range set id counts as decoder num_decoders.
 * d_counts (may be NULL): [num_decoders+1] queries per decoder.
 * d_tiles (may be NULL): [ntc_max_tiles(ctx, n)][3] = (decoder, first position
 * in perm, length) of every 128-query tile, in decoder order; d_num_tiles (may
 * be NULL): [1] the number of tiles written.  d_divergence (may be NULL): [2]
 * = { 1 if the query records were copied in bucket order, else 0;  the sum
 * over groups of 32 consecutive queries of (distinct decoders - 1), out-of-
 * range set ids counting as decoder num_decoders } -- Eq. 1's numerator; the
 * records are copied when that sum exceeds 4 x the number of groups.  Device
 * pointers; async. */
NTC_API ntc_status ntc_debug_bucket(ntc_ctx *ctx, const ntc_query *d_queries, size_t n, uint32_t *d_perm,
                            uint32_t *d_counts, uint32_t *d_tiles, uint32_t *d_num_tiles,
                            uint32_t *d_divergence, void *cuda_stream);

/* One query row as the default tensor-core decode (BUCKETED, TC_FP16/TC_BF16,
 * the standard shape) built it -- the bilinear fetch of Sec. 1's latent grids
 * that feeds x^_i = D_c(i)(z_i) of Sec. 3.3 -- recorded by
 * ntc_debug_decode_rows.  Level k, mip slot m (0: mip lo; 1: mip lo + 1,
 * written only when t > 0) and tap p in the order 00, 10, 01, 11:
 *   idx  texel index into `latents` (the ntc_desc array) of the tap, from the
 *        kernel's own texel coordinates;
 *   raw  the 16 bytes (8 fp16 channels) the kernel blended for the tap;
 *   w    the fp32 weight it blended them with: the bilinear weight times
 *        1 - t (slot 0 of a blend) or t (slot 1).  In clamp mode a row whose
 *        two texels coincide (an edge) carries the row's whole weight on tap
 *        0 (or 2) and weight 0 on tap 1 (or 3), whose raw is then unused;
 *   t, lo the mip pick;
 *   feat the MLP input as stored in tensor memory: 16 fp16 (TC_FP16) or bf16
 *        (TC_BF16) values, feat[i] holding inputs 2i (low half) and 2i + 1. */
typedef struct {
  uint64_t idx[2][2][4];
  uint32_t raw[2][2][4][4];
  float w[2][2][4];
  float t;
  uint32_t lo;
  uint32_t feat[8];
  uint32_t pad[6];
} ntc_debug_row; /* 512 bytes */

/* ntc_decode in BUCKETED mode through a debug instantiation of its tcgen05
 * kernel: the same bucketing, kernel template, launch configuration and
 * outputs (d_out as ntc_decode), and every good query's row recorded in
 * d_rows[i] (device array of n records; rows of bad queries are not
 * written).  TC_FP16/TC_BF16 contexts of the standard shape only
 * (NTC_ERR_UNSUPPORTED otherwise).  Device pointers; async. */
NTC_API ntc_status ntc_debug_decode_rows(ntc_ctx *ctx, const ntc_query *d_queries, size_t n, void *d_out,
                                         ntc_debug_row *d_rows, void *cuda_stream);

/* Upper bound on the number of 128-query tiles of n queries (no paper
 * counterpart). */
NTC_API size_t ntc_max_tiles(const ntc_ctx *ctx, size_t n);

/* Number of bad queries decoded since creation or the last reset (no paper
 * counterpart: the paper's queries are always valid).  Synchronises
 * the device.  Returns NTC_ERR_CUDA (and still writes *count) when a kernel
 * gave up one of its bounded waits since then (every mbarrier wait of the
 * tcgen05 kernels ends after 200 ms; the bucketing waits on nothing): that
 * call's results are invalid, the context stays usable.  The reset clears
 * both. */
NTC_API ntc_status ntc_get_error_count(ntc_ctx *ctx, uint64_t *count);
NTC_API ntc_status ntc_reset_error_count(ntc_ctx *ctx);

/* Test of the failure path above: one thread waits, with the decode kernels'
 * own bounded wait, for an mbarrier phase that nothing completes, gives up
 * after the 200 ms limit and records it in the context's status word exactly
 * as a decode kernel that gave up would.  Async on cuda_stream; nothing
 * faults, traps or hangs. */
NTC_API ntc_status ntc_debug_wait_timeout(ntc_ctx *ctx, void *cuda_stream);

/* Stage timing (no paper counterpart; Sec. 4.4 times whole kernels).  When
 * enabled, ntc_decode records CUDA events on its stream
 * before bucketing, between bucketing and the gather-decode, and after it.
 * ntc_stage_times waits for the last decode and returns, in milliseconds,
 * times[0] = bucketing (0 in divergent mode) and times[1] = gather-decode. */
NTC_API ntc_status ntc_set_stage_timing(ntc_ctx *ctx, int enable);
NTC_API ntc_status ntc_stage_times(ntc_ctx *ctx, float times[2]);

/* Kernels this context has launched since creation (host-side counter; no
 * paper counterpart). */
NTC_API uint64_t ntc_launch_count(const ntc_ctx *ctx);

/* ------------------------------------------------------ allocation-free entry
 *
 * The paper has no counterpart to this call; it exists for callers that may
 * not allocate device memory when they sort their queries -- for example a
 * renderer whose engine owns all GPU memory and forbids cudaMalloc and
 * cudaMallocAsync inside its frame loop, where an allocation can stall the
 * frame or fail half-way through it.
 *
 * ntc_bucket_static is the bucketing stage of ntc_debug_bucket without a
 * context and without any allocation: d_perm[n] receives the query indices in
 * (decoder, original index) order (out-of-range set ids count as decoder
 * num_decoders) and d_sorted[n] the query records in that order.  h_set_to_decoder
 * is a HOST array of num_sets entries (each < num_decoders); d_queries,
 * d_perm and d_sorted are caller-owned device buffers (the query buffers
 * 16-byte aligned).  Its kernels wait on nothing (no barrier, flag or
 * timeout), so a call that was enqueued completes.  Its scratch is one
 * file-scope device array of 2,409,472 bytes that every GPU loading the
 * library holds until the process exits, so:
 *   - num_sets <= 65536, num_decoders <= 4095 and
 *     (num_decoders + 1) * ceil(n / 2048) <= 262144 (larger calls return
 *     NTC_ERR_UNSUPPORTED and enqueue nothing);
 *   - every call on a device shares that array and it keeps the previous
 *     call's contents; the call clears what must start at zero itself, but two
 *     calls whose work overlaps on the GPU (different streams, threads or
 *     processes sharing the context) race and corrupt each other's result;
 *   - the first call on each device looks the array's device address up
 *     (cudaGetSymbolAddress) with that device current; make that first call
 *     before any stream capture.
 * Asynchronous on cuda_stream; n = 0 is a no-op.  It calls no cudaMalloc,
 * cudaFree or allocating library routine. */
NTC_API ntc_status ntc_bucket_static(const uint32_t *h_set_to_decoder, uint32_t num_sets,
                                     uint32_t num_decoders, const ntc_query *d_queries, size_t n,
                                     uint32_t *d_perm, ntc_query *d_sorted, void *cuda_stream);

/* ---------------------------------------------------------- map sources
 *
 * The clustered set -> decoder map of Alg. 2, Stage 2 (Sec. 3.3, "Clustering
 * into m groups"): k-means of the per-set embeddings (the paper uses 512-d CLIP
 * image features) into m groups; group g gets decoder g.  Lloyd's iteration in
 * fp64 on the current CUDA device:
 *   start       centroid g = h_features[h_init[g]] (m distinct rows < n, chosen
 *               by the caller, e.g. from a seeded permutation);
 *   assignment  c(i) = argmin_g sum_j (F[i][j] - mu_g[j])^2, the sum over j in
 *               increasing order, ties to the smallest g;
 *   update      mu_g = mean of the rows assigned to g, summed in increasing row
 *               order; an empty group keeps its centroid;
 *   stop        when no assignment changes, or after max_iters assignments.
 * Every fp64 operation is rounded to nearest without contraction, in that
 * order, so the result is reproducible bit for bit.
 * h_features: HOST [n][dim] fp32 (finite), 1 <= n <= 2^24, 1 <= dim <= 4096;
 * 1 <= m <= min(n, NTC_MAX_DECODERS).  Outputs (HOST, caller-owned): h_map[n]
 * = c(i) in [0, m); h_centroids (may be NULL) [m][dim] fp64, the means of the
 * final assignment; iters_run (may be NULL) the assignments made.
 * Synchronous; allocates and frees its own device memory. */
NTC_API ntc_status ntc_kmeans_map(const float *h_features, uint32_t n, uint32_t dim, uint32_t m,
                                  const uint32_t *h_init, uint32_t max_iters, uint32_t *h_map,
                                  double *h_centroids, uint32_t *iters_run);

/* Human-readable message of the last failed call on this host thread (no
 * paper counterpart). */
NTC_API const char *ntc_last_error(void);
NTC_API const char *ntc_status_string(ntc_status s);

#ifdef __cplusplus
}
#endif

#endif /* NTC_H */
