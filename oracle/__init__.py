"""CPU oracle for the runtime decode of neural-compressed textures.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  The product path (the
CUDA library and its Python binding) never imports, links or executes anything
here, and this package imports nothing from the product path.

What lives here:

* ``decode`` / ``taps`` / ``features`` -- thin ctypes wrappers around
  ``ntc_oracle.c`` (plain C, fp32 address math without contraction, double
  features and MLP).  The decode follows Sec. 3.3 (x^_i = D_{c(i)}(z_i)) and the
  decoder description of Sec. 4 (3-layer MLP, first two layers hidden); the
  sampling rule the paper leaves open is written out in the C file's header.
* ``bucket`` -- the stable counting sort of queries by decoder id that the
  paper's divergence argument (Sec. 2) motivates: ``perm`` lists query indices in
  (decoder, original index) order, with a numpy stable argsort as the library
  step; ``counts``/``offsets`` are its histogram and exclusive scan, ``tiles``
  the consecutive 128-query chunks of each decoder's segment.
* ``divergence_map`` / ``divergence_score`` -- the divergence map D of Sec. 2
  (number of distinct ids per block) and the score of Eq. 1 (mean |D - 1|).
* ``speedup_percent`` -- the reading of the "average speedup" figures printed
  under Tables 5 and 6: mean over resolutions of (t_baseline / t_shared - 1).
* ``kmeans`` -- Alg. 2 Stage 2: k-means over per-texture embeddings into m
  groups (the set -> decoder map c(i)); Lloyd's iteration in double, written
  out in ``ntc_oracle.c`` with the start, tie and empty-group rules it uses.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ntc_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libntc_oracle.so")
_lock = threading.Lock()
_lib = None

QUERY_DTYPE = np.dtype([("set_id", "<u4"), ("u", "<f4"), ("v", "<f4"), ("lod", "<f4")])
TILE_ROWS = 128


def build(force: bool = False) -> str:
    """Compile ntc_oracle.c with gcc (no FMA contraction, IEEE semantics)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-pthread",
               "-ffp-contract=off", "-fno-fast-math", "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class _Assets(ctypes.Structure):
    _fields_ = [
        ("num_sets", ctypes.c_uint32),
        ("num_levels", ctypes.c_uint32),
        ("num_mips", ctypes.c_uint32),
        ("channels", ctypes.c_uint32),
        ("level_dims", ctypes.c_void_p),
        ("latent_offsets", ctypes.c_void_p),
        ("latents", ctypes.c_void_p),
        ("address_mode", ctypes.c_uint32),
        ("num_decoders", ctypes.c_uint32),
        ("in_dim", ctypes.c_uint32),
        ("hidden", ctypes.c_uint32),
        ("num_hidden_layers", ctypes.c_uint32),
        ("out_dim", ctypes.c_uint32),
        ("weights", ctypes.c_void_p),
        ("set_to_decoder", ctypes.c_void_p),
        ("pe_frequencies", ctypes.c_uint32),
        ("activation", ctypes.c_uint32),
        ("leaky_slope", ctypes.c_float),
    ]


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            lib.or_param_count.argtypes = [P]
            lib.or_param_count.restype = ctypes.c_size_t
            lib.or_taps.argtypes = [P, P, ctypes.c_size_t, P, P, P]
            lib.or_taps.restype = None
            lib.or_features.argtypes = [P, P, ctypes.c_size_t, P]
            lib.or_features.restype = None
            lib.or_decode.argtypes = [P, P, ctypes.c_size_t, P, ctypes.c_int]
            lib.or_decode.restype = ctypes.c_uint64
            U = ctypes.c_uint32
            lib.or_kmeans.argtypes = [P, U, U, U, P, U, P, P]
            lib.or_kmeans.restype = U
            _lib = lib
    return _lib


def _c(arr, dtype):
    a = np.ascontiguousarray(arr, dtype=dtype)
    return a


class _Bound:
    """ctypes view of an assets object; keeps the numpy buffers alive."""

    def __init__(self, a):
        self.keep = [
            _c(a.level_dims, np.uint32),
            _c(a.latent_offsets, np.uint64),
            _c(a.latents, np.uint16),
            _c(a.weights, np.float32),
            _c(a.set_to_decoder, np.uint32),
        ]
        dims, offs, lat, w, m = self.keep
        if a.channels > 64:
            raise ValueError("oracle supports at most 64 channels per texel")
        self.s = _Assets(
            a.num_sets, a.num_levels, a.num_mips, a.channels,
            dims.ctypes.data, offs.ctypes.data, lat.ctypes.data, a.address_mode,
            a.num_decoders, a.in_dim, a.hidden, a.num_hidden_layers, a.out_dim,
            w.ctypes.data, m.ctypes.data, getattr(a, "pe_frequencies", 0), getattr(a, "activation", 0),
            getattr(a, "leaky_slope", 0.0))
        lib = _load()
        per = lib.or_param_count(ctypes.byref(self.s))
        if w.size != per * a.num_decoders:
            raise ValueError(f"weights hold {w.size} values, expected {per} x {a.num_decoders}")
        if a.in_dim != a.num_levels * a.channels + 4 * getattr(a, "pe_frequencies", 0):
            raise ValueError("in_dim must equal num_levels * channels + 4 * pe_frequencies")

    @property
    def ptr(self):
        return ctypes.byref(self.s)


def _queries(q) -> np.ndarray:
    q = np.ascontiguousarray(q)
    if q.dtype.itemsize != 16:
        raise ValueError("queries must be 16-byte records (set_id, u, v, lod)")
    return q.view(QUERY_DTYPE).reshape(-1)


def param_count(assets) -> int:
    return int(_load().or_param_count(_Bound(assets).ptr))


def decode(assets, queries, nthreads: int | None = None):
    """Decoded texels, float64 [n][out_dim], and the number of bad queries."""
    b = _Bound(assets)
    q = _queries(queries)
    out = np.empty((q.shape[0], assets.out_dim), dtype=np.float64)
    nt = nthreads or os.cpu_count() or 1
    bad = _load().or_decode(b.ptr, q.ctypes.data, q.shape[0], out.ctypes.data, nt)
    return out, int(bad)


def taps(assets, queries):
    """Texel indices u64 [n][L][2][4], fp32 weights [n][L][2][4] and blend t [n]."""
    b = _Bound(assets)
    q = _queries(queries)
    n, L = q.shape[0], assets.num_levels
    idx = np.empty((n, L, 2, 4), dtype=np.uint64)
    w = np.empty((n, L, 2, 4), dtype=np.float32)
    t = np.empty((n,), dtype=np.float32)
    _load().or_taps(b.ptr, q.ctypes.data, n, idx.ctypes.data, w.ctypes.data, t.ctypes.data)
    return idx, w, t


def features(assets, queries):
    """MLP inputs, float64 [n][in_dim] (NaN rows for bad queries)."""
    b = _Bound(assets)
    q = _queries(queries)
    f = np.empty((q.shape[0], assets.in_dim), dtype=np.float64)
    _load().or_features(b.ptr, q.ctypes.data, q.shape[0], f.ctypes.data)
    return f


def decoder_ids(set_ids, set_to_decoder, num_decoders):
    """Decoder id per query; a set id outside the map goes to bucket num_decoders."""
    s = np.asarray(set_ids, dtype=np.uint64)
    m = np.asarray(set_to_decoder, dtype=np.uint32)
    ok = s < m.shape[0]
    d = np.full(s.shape, num_decoders, dtype=np.uint32)
    d[ok] = m[s[ok].astype(np.int64)]
    return d


def bucket(set_ids, set_to_decoder, num_decoders, tile_rows: int = TILE_ROWS):
    """Stable counting sort by decoder id.

    Returns ``perm`` (u32 [n]: query indices in (decoder, index) order),
    ``counts`` and ``offsets`` (u32 [num_decoders + 1], the last bucket holding
    queries whose set id is out of range) and ``tiles`` (u32 [T][3]: decoder,
    first position in perm, length), the consecutive ``tile_rows`` chunks of each
    decoder's segment in decoder order.
    """
    d = decoder_ids(set_ids, set_to_decoder, num_decoders)
    perm = np.argsort(d, kind="stable").astype(np.uint32)
    counts = np.bincount(d, minlength=num_decoders + 1).astype(np.uint64)
    offsets = np.zeros_like(counts)
    offsets[1:] = np.cumsum(counts)[:-1]
    tiles = []
    for dec in range(num_decoders + 1):
        c, o = int(counts[dec]), int(offsets[dec])
        for s in range(0, c, tile_rows):
            tiles.append((dec, o + s, min(tile_rows, c - s)))
    tiles = np.array(tiles, dtype=np.uint32).reshape(-1, 3)
    return perm, counts.astype(np.uint32), offsets.astype(np.uint32), tiles


def divergence_map(ids, block: int = 32):
    """D of Sec. 2: number of distinct ids in each block of ``block`` consecutive
    entries of ``ids`` (the last block may be partial)."""
    ids = np.asarray(ids)
    nb = (ids.shape[0] + block - 1) // block
    return np.array([len(set(ids[b * block:(b + 1) * block].tolist())) for b in range(nb)],
                    dtype=np.int64)


def divergence_score(X):
    """Eq. 1: the mean of |X_ij - 1| over all entries of the divergence map X."""
    X = np.asarray(X, dtype=np.float64)
    return float(np.mean(np.abs(X - 1.0)))


def speedup_percent(t_baseline, t_shared):
    """Average speedup as printed under Tables 5-6: 100 * mean(t_b / t_s - 1)."""
    tb = np.asarray(t_baseline, dtype=np.float64)
    ts = np.asarray(t_shared, dtype=np.float64)
    return float(100.0 * np.mean(tb / ts - 1.0))


def kmeans(features, m: int, init, max_iters: int = 100):
    """Alg. 2, Stage 2: k-means of the rows of ``features`` [n, dim] (fp32) into
    ``m`` groups, starting from the rows ``init`` (m distinct indices).
    Returns (map [n] uint32, centroids [m, dim] float64, assignments made)."""
    F = np.ascontiguousarray(features, dtype=np.float32)
    n, dim = F.shape
    init = np.ascontiguousarray(init, dtype=np.uint32)
    if init.shape != (m,) or len(set(init.tolist())) != m or (init >= n).any():
        raise ValueError("init must hold m distinct row indices")
    out = np.empty(n, dtype=np.uint32)
    mu = np.empty((m, dim), dtype=np.float64)
    it = _load().or_kmeans(F.ctypes.data, n, dim, m, init.ctypes.data, max_iters, out.ctypes.data,
                           mu.ctypes.data)
    return out, mu, int(it)
