"""Seeded synthetic workloads for the neural-texture decode.

The paper's datasets (Polyhaven textures, the Yokohama/Bistro/ToyShop scenes)
and its trained weights are not available, so every input here is synthetic with
the shapes of the paper's workloads: 1k-2k textures, 1-512 texture sets, one
decoder per set, per cluster or shared by all (Sec. 3.1, Sec. 4), queries
interleaved as a rendering pass emits them (Sec. 2).

This module generates inputs only; it holds none of the decode arithmetic.  The
heavy lifting (normals, mip chains, Voronoi labelling) is ``gen.c``, compiled
with gcc on first use.  Both the CUDA library and the CPU oracle consume the
arrays built here.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "gen.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libntcgen.so")
_lock = threading.Lock()
_lib = None

QUERY_DTYPE = np.dtype([("set_id", "<u4"), ("u", "<f4"), ("v", "<f4"), ("lod", "<f4")])
BASE_SEED = 260827888
SIGMA = 0.5  # standard deviation of the latent values


def build(force: bool = False) -> str:
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-pthread",
                        "-ffp-contract=off", "-o", tmp, _SRC, "-lm"], check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P, U32, U64, I = ctypes.c_void_p, ctypes.c_uint32, ctypes.c_uint64, ctypes.c_int
            lib.gen_key.argtypes = [U64, U64, U64, U64]
            lib.gen_key.restype = U64
            lib.gen_double_to_half.argtypes = [ctypes.c_double]
            lib.gen_double_to_half.restype = ctypes.c_uint16
            lib.gen_latents.argtypes = [U64, U32, U32, U32, U32, P, P, ctypes.c_double, P, I]
            lib.gen_decoder.argtypes = [U64, U32, U32, U32, U32, U32, P]
            lib.gen_permutation.argtypes = [U64, U64, U32, P]
            lib.gen_queries_uniform.argtypes = [U64, U64, U32, P]
            lib.gen_queries_texel_centres.argtypes = [U32, U32, P]
            lib.gen_queries_controlled.argtypes = [U64, U32, U32, U32, P]
            lib.gen_gbuffer.argtypes = [U64, U32, U32, U32, U32, U32, U32, I, ctypes.c_float, P, P, I]
            for f in ("gen_latents", "gen_decoder", "gen_permutation", "gen_queries_uniform",
                      "gen_queries_texel_centres", "gen_queries_controlled", "gen_gbuffer"):
                getattr(lib, f).restype = None
            _lib = lib
    return _lib


def _threads() -> int:
    return max(1, os.cpu_count() or 1)


@dataclasses.dataclass
class Assets:
    """Everything ``ntc_create`` consumes (host arrays)."""
    num_sets: int
    num_levels: int
    num_mips: int
    channels: int
    level_dims: np.ndarray       # u32 [S][L][2]  (W, H of mip 0)
    latent_offsets: np.ndarray   # u64 [S][L][M]  texel offsets into latents
    latents: np.ndarray          # u16 [texels * channels]  (IEEE half bits)
    num_decoders: int
    in_dim: int
    hidden: int
    num_hidden_layers: int
    out_dim: int
    weights: np.ndarray          # f32 [D][params]
    set_to_decoder: np.ndarray   # u32 [S]
    address_mode: int = 0        # 0 wrap, 1 clamp
    pe_frequencies: int = 0      # F: 4F positional-encoding inputs after the latents
    activation: int = 0          # 0 ReLU, 1 LeakyReLU
    leaky_slope: float = 0.01    # LeakyReLU slope (the PyTorch default)

    @property
    def params_per_decoder(self) -> int:
        H, I, C = self.hidden, self.in_dim, self.out_dim
        return H * I + H + (self.num_hidden_layers - 1) * (H * H + H) + C * H + C

    @property
    def latent_bytes(self) -> int:
        return int(self.latents.nbytes)


@dataclasses.dataclass
class Workload:
    name: str
    assets: Assets
    queries: np.ndarray          # QUERY_DTYPE [n]
    info: dict


def pyramid_layout(num_sets, level_dims, num_mips):
    """Texel offsets [S][L][M] of a packed set-major, level-major, mip-major layout."""
    dims = np.asarray(level_dims, dtype=np.uint32).reshape(num_sets, -1, 2)
    L = dims.shape[1]
    offs = np.zeros((num_sets, L, num_mips), dtype=np.uint64)
    cur = 0
    for s in range(num_sets):
        for k in range(L):
            W, H = int(dims[s, k, 0]), int(dims[s, k, 1])
            for m in range(num_mips):
                offs[s, k, m] = cur
                cur += max(1, W >> m) * max(1, H >> m)
    return dims, offs, cur


def make_latents(seed, num_sets, level_dims, num_mips, channels=8, sigma=SIGMA):
    dims, offs, total = pyramid_layout(num_sets, level_dims, num_mips)
    lat = np.empty(total * channels, dtype=np.uint16)
    _load().gen_latents(seed, num_sets, dims.shape[1], num_mips, channels,
                        dims.ctypes.data, offs.ctypes.data, sigma, lat.ctypes.data, _threads())
    return dims, offs, lat


def make_weights(seed, num_decoders, in_dim, hidden, layers, out_dim):
    per = hidden * in_dim + hidden + (layers - 1) * (hidden * hidden + hidden) + out_dim * hidden + out_dim
    w = np.empty((num_decoders, per), dtype=np.float32)
    lib = _load()
    for d in range(num_decoders):
        lib.gen_decoder(seed, d, in_dim, hidden, layers, out_dim, w[d].ctypes.data)
    return w


def permutation(seed, tag, n):
    p = np.empty(n, dtype=np.uint32)
    _load().gen_permutation(seed, tag, n, p.ctypes.data)
    return p


def map_identity(num_sets):
    return np.arange(num_sets, dtype=np.uint32)


def map_shared(num_sets):
    return np.zeros(num_sets, dtype=np.uint32)


def map_random_partition(seed, num_sets, num_decoders, tag=0):
    """Balanced seeded partition: the i-th set of a seeded permutation goes to
    decoder i mod num_decoders (group sizes differ by at most one)."""
    p = permutation(seed, 100 + tag, num_sets)
    m = np.empty(num_sets, dtype=np.uint32)
    m[p] = np.arange(num_sets, dtype=np.uint32) % num_decoders
    return m


# Textures per category of the paper's 586-texture evaluation set (Table 1):
# Aerial, Brick, Concrete, Fabric, Floor, Metal, Plaster/Concrete, Rock,
# Roofing, Terrain, Wood.
CATEGORY_SIZES = (20, 80, 40, 37, 123, 24, 19, 50, 21, 107, 65)


def map_category(sizes=CATEGORY_SIZES):
    """Category grouping (Sec. 4.1, "Category"): the first sizes[0] sets go to
    decoder 0, the next sizes[1] to decoder 1, and so on."""
    return np.repeat(np.arange(len(sizes), dtype=np.uint32), np.asarray(sizes, dtype=np.int64))


def map_random_sizes(seed, sizes, tag=0):
    """Random grouping with prescribed group sizes (Sec. 4.1, "Random": the same
    group sizes as another grouping): a seeded permutation of map_category."""
    m = map_category(sizes)
    p = permutation(seed, 200 + tag, len(m))
    out = np.empty_like(m)
    out[p] = m
    return out


def group_sizes(set_to_decoder, num_decoders):
    return np.bincount(np.asarray(set_to_decoder, dtype=np.int64), minlength=num_decoders)


def embeddings(seed, sizes, dim=512, spread=0.8):
    """Synthetic stand-in for the per-texture CLIP image embeddings of Alg. 2
    (Stage 1, 512-d): group g (sizes[g] sets, in map_category order) has a random
    unit centre; each set's embedding is its centre plus isotropic noise of norm
    about `spread`, normalised to unit length (CLIP features are compared on the
    unit sphere).  fp32 [sum(sizes), dim]."""
    rng = np.random.default_rng(seed)
    k = len(sizes)
    c = rng.standard_normal((k, dim))
    c /= np.linalg.norm(c, axis=1, keepdims=True)
    lab = map_category(sizes)
    x = c[lab] + spread * rng.standard_normal((len(lab), dim)) / np.sqrt(dim)
    x /= np.linalg.norm(x, axis=1, keepdims=True)
    return x.astype(np.float32)


def kmeans_init(seed, n, m, tag=0):
    """m distinct start rows for k-means: the first m of a seeded permutation."""
    return permutation(seed, 300 + tag, n)[:m].copy()


def queries_uniform(seed, n, num_sets):
    q = np.empty(n, dtype=QUERY_DTYPE)
    _load().gen_queries_uniform(seed, n, num_sets, q.ctypes.data)
    return q


def queries_texel_centres(N, set_id=0):
    q = np.empty(N * N, dtype=QUERY_DTYPE)
    _load().gen_queries_texel_centres(N, set_id, q.ctypes.data)
    return q


def queries_controlled(seed, N, num_sets, d):
    if not (1 <= d <= 32 and d <= num_sets and N % 8 == 0):
        raise ValueError("need 1 <= d <= min(32, num_sets) and N % 8 == 0")
    q = np.empty(N * N, dtype=QUERY_DTYPE)
    _load().gen_queries_controlled(seed, N, num_sets, d, q.ctypes.data)
    return q


def queries_gbuffer(seed, width, height, regions, num_sets, T, lod_mode=0, lod_max=3.0,
                    frames=1, with_labels=False):
    if width % 8 or height % 4 or regions < 1:
        raise ValueError("screen must be a whole number of 8x4 tiles, regions >= 1")
    n = width * height
    q = np.empty(n * frames, dtype=QUERY_DTYPE)
    lab = np.empty(n * frames, dtype=np.uint32) if with_labels else None
    lib = _load()
    for f in range(frames):
        lib.gen_gbuffer(seed, f, width, height, regions, num_sets, T, lod_mode, lod_max,
                        q[f * n:].ctypes.data, lab[f * n:].ctypes.data if with_labels else None,
                        _threads())
    return (q, lab) if with_labels else q


def make_assets(seed, num_sets, T, num_mips, num_decoders, set_to_decoder, hidden=64,
                out_dim=8, layers=2, channels=8, address_mode=0, levels=2, pe_frequencies=0,
                activation=0, leaky_slope=0.01, grid=None):
    """Latent levels per set: two (L0 at T/2, L1 at T/4, square) or one; `grid`
    overrides the size of a single level (the paper's 256^2 grid)."""
    sizes = [(T // 2, T // 2), (T // 4, T // 4)][:levels] if grid is None else [(grid, grid)]
    dims = [sizes for _ in range(num_sets)]
    dims, offs, lat = make_latents(seed, num_sets, dims, num_mips, channels)
    L = dims.shape[1]
    in_dim = L * channels + 4 * pe_frequencies
    w = make_weights(seed, num_decoders, in_dim, hidden, layers, out_dim)
    return Assets(num_sets=num_sets, num_levels=L, num_mips=num_mips, channels=channels,
                  level_dims=dims, latent_offsets=offs, latents=lat,
                  num_decoders=num_decoders, in_dim=in_dim, hidden=hidden,
                  num_hidden_layers=layers, out_dim=out_dim, weights=w,
                  set_to_decoder=np.asarray(set_to_decoder, dtype=np.uint32),
                  address_mode=address_mode, pe_frequencies=pe_frequencies,
                  activation=activation, leaky_slope=leaky_slope)


# --------------------------------------------------------------- named workloads
#
# full  = the sizes of the five workloads:
#   raster-256                  one 256^2 set, one decoder, a texel-centre raster;
#   uniform-4m                  16 sets of 1024^2, a decoder per set, 4,194,304
#                               queries with uniform set id and UV;
#   gbuffer-1080p               a 1920x1080 G-buffer over 32 sets of 1024^2 (4 mips);
#   gbuffer-2160p               a 3840x2160 G-buffer over 128 sets of 2048^2;
#   gbuffer-2160p-x4-trilinear  4 frames of 3840x2160 over 512 sets of 2048^2,
#                               16->128->128->9 decoders, continuous lods;
# small = the same recipes shrunk so the oracle finishes in seconds, still
#         spanning many 128-query tiles and a ragged tail.
# medium (gbuffer-2160p-x4-trilinear only) = one frame over 32 of the sets,
#         about 3 GB on the device: the size of a full ncu capture.

# seed offset of each named workload (the generated inputs depend on it)
_SEED = {"raster-256": 1, "uniform-4m": 2, "gbuffer-1080p": 3, "gbuffer-2160p": 4,
         "gbuffer-2160p-x4-trilinear": 5}
WORKLOADS = tuple(_SEED)


def named(name: str, size: str = "full", variant: str | None = None, query_tag: int = 0) -> Workload:
    """One of WORKLOADS.  variant: the set->decoder grouping of gbuffer-1080p
    ("identity", "clustered4", "shared") or the decoder count of gbuffer-2160p
    ("128", "16", "8", "1").  query_tag != 0 draws another query stream of the
    same recipe over the same assets (one per rank of a multi-GPU run)."""
    if name not in _SEED:
        raise ValueError(f"unknown workload {name}")
    seed = BASE_SEED + _SEED[name]
    if query_tag:
        w = named(name, size, variant)
        qseed = seed + 1000 * query_tag
        if name == "raster-256":
            return w  # a raster of texel centres has only one query stream
        if name == "uniform-4m":
            q = queries_uniform(qseed, len(w.queries), w.assets.num_sets)
        else:
            W_, H_, R, F = {("gbuffer-1080p", True): (1920, 1080, 200, 1), ("gbuffer-1080p", False): (240, 136, 40, 1),
                            ("gbuffer-2160p", True): (3840, 2160, 800, 1), ("gbuffer-2160p", False): (320, 180, 120, 1),
                            ("gbuffer-2160p-x4-trilinear", True): (3840, 2160, 2000, 4),
                            ("gbuffer-2160p-x4-trilinear", False): (256, 128, 60, 2)}[(name, size == "full")]
            tri = name == "gbuffer-2160p-x4-trilinear"
            q = queries_gbuffer(qseed, W_, H_, R, w.assets.num_sets, w.info["T"], lod_mode=1 if tri else 0,
                                lod_max=3.0, frames=F)
        return Workload(f"{w.name}-q{query_tag}", w.assets, q, dict(w.info, query_tag=query_tag))
    full = size == "full"
    if name == "raster-256":
        T = 256 if full else 64
        a = make_assets(seed, 1, T, 1, 1, map_shared(1))
        q = queries_texel_centres(T, 0)
        return Workload(f"{name}-{size}", a, q, {"T": T, "maps": "shared"})
    if name == "uniform-4m":
        S, T, n = (16, 1024, 4_194_304) if full else (16, 128, 40_000 + 77)
        a = make_assets(seed, S, T, 1, S, map_identity(S))
        q = queries_uniform(seed, n, S)
        return Workload(f"{name}-{size}", a, q, {"T": T, "maps": "identity"})
    if name == "gbuffer-1080p":
        S, T = 32, (1024 if full else 128)
        W, H, R = (1920, 1080, 200) if full else (240, 136, 40)
        variant = variant or "identity"
        m = {"identity": map_identity(S), "clustered4": map_random_partition(seed, S, 4),
             "shared": map_shared(S)}[variant]
        D = {"identity": S, "clustered4": 4, "shared": 1}[variant]
        a = make_assets(seed, S, T, 4, D, m)
        q = queries_gbuffer(seed, W, H, R, S, T, lod_mode=0)
        return Workload(f"{name}-{size}-{variant}", a, q, {"T": T, "maps": variant})
    if name == "gbuffer-2160p":
        S, T = (128, 2048) if full else (128, 64)
        W, H, R = (3840, 2160, 800) if full else (320, 180, 120)
        D = int(variant or 128)
        m = map_identity(S) if D == S else map_random_partition(seed, S, D)
        a = make_assets(seed, S, T, 4, D, m, out_dim=9)
        q = queries_gbuffer(seed, W, H, R, S, T, lod_mode=0)
        return Workload(f"{name}-{size}-{D}", a, q, {"T": T, "maps": f"random{D}"})
    if size == "medium":  # the profiling size: same grids, decoders and screen, 32 sets, one frame
        S, T, (W, H, R, F) = 32, 2048, (3840, 2160, 2000, 1)
    else:
        S, T = (512, 2048) if full else (24, 128)
        W, H, R, F = (3840, 2160, 2000, 4) if full else (256, 128, 60, 2)
    D = 8
    a = make_assets(seed, S, T, 4, D, map_random_partition(seed, S, D), hidden=128, out_dim=9)
    q = queries_gbuffer(seed, W, H, R, S, T, lod_mode=1, lod_max=3.0, frames=F)
    return Workload(f"{name}-{size}", a, q, {"T": T, "maps": "random8", "frames": F})


def paper_decoder(size: str = "full", hidden=64, layers=2, levels=1, channels=4, pe=4, activation=1,
                  leaky_slope=0.01, num_sets=16, num_decoders=4, out_dim=9, trilinear=True) -> Workload:
    """The decoder of the paper's experiments (Sec. 4): one 256x256x4 latent grid
    per set (64^2 small) with a 4-level mip chain, its bilinear (trilinear when
    the lod is fractional) features concatenated with a positional encoding of
    `pe` frequencies, an MLP of `layers` hidden layers of `hidden` neurons with
    LeakyReLU (the A x B ablation varies both), sigmoid output; the sets grouped
    into `num_decoders` clusters.  Queries: a 1920x1080 G-buffer (240x136
    small) with 200 (40) regions and a continuous lod in [0, 3] per region."""
    full = size == "full"
    seed = BASE_SEED + 40 + hidden + 7 * layers + levels + channels + pe + activation
    grid = 256 if full else 64
    W_, H_, R = (1920, 1080, 200) if full else (240, 136, 40)
    m = map_random_partition(seed, num_sets, num_decoders)
    a = make_assets(seed, num_sets, 2 * grid, 4, num_decoders, m, hidden=hidden, out_dim=out_dim,
                    layers=layers, channels=channels, levels=levels, pe_frequencies=pe,
                    activation=activation, leaky_slope=leaky_slope, grid=grid if levels == 1 else None)
    q = queries_gbuffer(seed, W_, H_, R, num_sets, grid, lod_mode=1 if trilinear else 0, lod_max=3.0)
    name = f"paper-A{hidden}xB{layers + 1}-L{levels}C{channels}F{pe}{'leaky' if activation else 'relu'}-{size}"
    return Workload(name, a, q, {"grid": grid})


def sweep(d: int, N: int = 4096, size: str = "full") -> Workload:
    """Controlled-divergence sweep: 32 sets of 1024^2 (128^2 small), 32 decoders,
    identity map, N x N texel-centre raster, exactly d distinct sets per warp."""
    S, T = 32, (1024 if size == "full" else 128)
    seed = BASE_SEED + 100
    a = make_assets(seed, S, T, 1, S, map_identity(S))
    q = queries_controlled(seed + d, N, S, d)
    return Workload(f"sweep-d{d}-N{N}", a, q, {"d": d, "N": N, "T": T})
