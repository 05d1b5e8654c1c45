"""Python binding of libntc (``include/ntc.h``): ctypes marshalling only.

The module-level ``ntc_*`` functions mirror the C ABI one to one and take raw
pointers (ints) and sizes.  ``Decoder`` wraps them for torch tensors: PyTorch
supplies device memory and streams, every step of the decode runs in libntc's
CUDA kernels.  There is no fallback: if ``_build/libntc.so`` is missing the
import of this module fails.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libntc.so")

NTC_OK, NTC_ERR_INVALID_ARG, NTC_ERR_UNSUPPORTED, NTC_ERR_OUT_OF_MEMORY, NTC_ERR_CUDA = range(5)
NTC_PREC_TC_FP16, NTC_PREC_TC_BF16, NTC_PREC_FP32 = range(3)
NTC_MODE_BUCKETED, NTC_MODE_DIVERGENT, NTC_MODE_BUCKETED_MMA, NTC_MODE_DIVERGENT_FMA = range(4)
NTC_MAX_DECODERS = 4095
NTC_TILE_ROWS = 128

# ntc_debug_row (include/ntc.h), 512 bytes
DEBUG_ROW = np.dtype([("idx", "<u8", (2, 2, 4)), ("raw", "<u4", (2, 2, 4, 4)), ("w", "<f4", (2, 2, 4)),
                      ("t", "<f4"), ("lo", "<u4"), ("feat", "<u4", (8,)), ("pad", "<u4", (6,))])
assert DEBUG_ROW.itemsize == 512

PRECISIONS = {"fp16": NTC_PREC_TC_FP16, "bf16": NTC_PREC_TC_BF16, "fp32": NTC_PREC_FP32}
NTC_OUTPUT_FP32, NTC_OUTPUT_FP16 = 0, 1
OUTPUTS = {"fp32": NTC_OUTPUT_FP32, "fp16": NTC_OUTPUT_FP16}
MODES = {"bucketed": NTC_MODE_BUCKETED, "divergent": NTC_MODE_DIVERGENT, "bucketed_mma": NTC_MODE_BUCKETED_MMA,
         "divergent_fma": NTC_MODE_DIVERGENT_FMA}
EXPORTS = ("ntc_create", "ntc_decode", "ntc_decode_host", "ntc_destroy", "ntc_debug_taps", "ntc_debug_decode_rows",
           "ntc_debug_features", "ntc_debug_bucket", "ntc_max_tiles", "ntc_get_error_count",
           "ntc_reset_error_count", "ntc_launch_count", "ntc_set_stage_timing", "ntc_stage_times",
           "ntc_bucket_static", "ntc_kmeans_map", "ntc_debug_wait_timeout", "ntc_last_error",
           "ntc_status_string")


class ntc_desc(ctypes.Structure):
    _fields_ = [
        ("num_sets", ctypes.c_uint32),
        ("num_decoders", ctypes.c_uint32),
        ("latent_channels", ctypes.c_uint32),
        ("num_levels", ctypes.c_uint32),
        ("num_mips", ctypes.c_uint32),
        ("level_dims", ctypes.c_void_p),
        ("latent_offsets", ctypes.c_void_p),
        ("latents", ctypes.c_void_p),
        ("num_texels", ctypes.c_uint64),
        ("in_dim", ctypes.c_uint32),
        ("hidden", ctypes.c_uint32),
        ("num_hidden_layers", ctypes.c_uint32),
        ("out_dim", ctypes.c_uint32),
        ("weights", ctypes.c_void_p),
        ("set_to_decoder", ctypes.c_void_p),
        ("precision", ctypes.c_int),
        ("address_mode", ctypes.c_uint32),
        ("pe_frequencies", ctypes.c_uint32),
        ("activation", ctypes.c_uint32),
        ("leaky_slope", ctypes.c_float),
        ("output_format", ctypes.c_uint32),
    ]


class NtcError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"{msg} (status {status})")
        self.status = status


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"libntc is not built ({LIB_PATH} missing); run __graft_entry__.build()")
    lib = ctypes.CDLL(LIB_PATH)
    P, S, I = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int
    sig = {
        "ntc_create": ([P, P], I),
        "ntc_decode": ([P, P, S, P, P, I], I),
        "ntc_decode_host": ([P, P, S, P, P, I], I),
        "ntc_destroy": ([P], I),
        "ntc_debug_taps": ([P, P, S, P, P, P, P], I),
        "ntc_debug_features": ([P, P, S, P, P], I),
        "ntc_debug_decode_rows": ([P, P, S, P, P, P], I),
        "ntc_debug_bucket": ([P, P, S, P, P, P, P, P, P], I),
        "ntc_max_tiles": ([P, S], S),
        "ntc_get_error_count": ([P, P], I),
        "ntc_reset_error_count": ([P], I),
        "ntc_debug_wait_timeout": ([P, P], I),
        "ntc_launch_count": ([P], ctypes.c_uint64),
        "ntc_set_stage_timing": ([P, I], I),
        "ntc_stage_times": ([P, P], I),
        "ntc_bucket_static": ([P, ctypes.c_uint32, ctypes.c_uint32, P, S, P, P, P], I),
        "ntc_kmeans_map": ([P, ctypes.c_uint32, ctypes.c_uint32, ctypes.c_uint32, P, ctypes.c_uint32, P, P, P], I),
        "ntc_last_error": ([], ctypes.c_char_p),
        "ntc_status_string": ([I], ctypes.c_char_p),
    }
    for name, (args, res) in sig.items():
        f = getattr(lib, name)
        f.argtypes = args
        f.restype = res
    return lib


_lib = _load()


def _check(status):
    if status != NTC_OK:
        raise NtcError(status, _lib.ntc_last_error().decode())


# ------------------------------------------------------- 1:1 mirrors of the ABI

def ntc_create(desc: ntc_desc) -> int:
    ctx = ctypes.c_void_p()
    _check(_lib.ntc_create(ctypes.byref(desc), ctypes.byref(ctx)))
    return ctx.value


def ntc_decode(ctx, d_queries, n, d_out, stream, mode):
    _check(_lib.ntc_decode(ctx, d_queries, n, d_out, stream, mode))


def ntc_decode_host(ctx, h_queries, n, h_out, stream, mode):
    _check(_lib.ntc_decode_host(ctx, h_queries, n, h_out, stream, mode))


def ntc_destroy(ctx):
    _check(_lib.ntc_destroy(ctx))


def ntc_debug_taps(ctx, d_queries, n, d_idx, d_w, d_t, stream):
    _check(_lib.ntc_debug_taps(ctx, d_queries, n, d_idx, d_w, d_t, stream))


def ntc_debug_features(ctx, d_queries, n, d_feat, stream):
    _check(_lib.ntc_debug_features(ctx, d_queries, n, d_feat, stream))


def ntc_debug_decode_rows(ctx, d_queries, n, d_out, d_rows, stream):
    _check(_lib.ntc_debug_decode_rows(ctx, d_queries, n, d_out, d_rows, stream))


def ntc_debug_bucket(ctx, d_queries, n, d_perm, d_counts, d_tiles, d_num_tiles, d_divergence, stream):
    _check(_lib.ntc_debug_bucket(ctx, d_queries, n, d_perm, d_counts, d_tiles, d_num_tiles, d_divergence,
                                 stream))


def ntc_max_tiles(ctx, n) -> int:
    return int(_lib.ntc_max_tiles(ctx, n))


def ntc_get_error_count(ctx) -> int:
    v = ctypes.c_uint64()
    _check(_lib.ntc_get_error_count(ctx, ctypes.byref(v)))
    return int(v.value)


def ntc_reset_error_count(ctx):
    _check(_lib.ntc_reset_error_count(ctx))


def ntc_debug_wait_timeout(ctx, stream=None):
    _check(_lib.ntc_debug_wait_timeout(ctx, stream))


def ntc_launch_count(ctx) -> int:
    return int(_lib.ntc_launch_count(ctx))


def ntc_set_stage_timing(ctx, enable):
    _check(_lib.ntc_set_stage_timing(ctx, int(bool(enable))))


def ntc_stage_times(ctx):
    t = (ctypes.c_float * 2)()
    _check(_lib.ntc_stage_times(ctx, t))
    return float(t[0]), float(t[1])


def ntc_bucket_static(h_set_to_decoder, num_sets, num_decoders, d_queries, n, d_perm, d_sorted, stream):
    """Allocation-free bucketing (no context): see include/ntc.h."""
    _check(_lib.ntc_bucket_static(h_set_to_decoder, num_sets, num_decoders, d_queries, n, d_perm,
                                  d_sorted, stream))


def ntc_kmeans_map(h_features, n, dim, m, h_init, max_iters, h_map, h_centroids, iters_run):
    _check(_lib.ntc_kmeans_map(h_features, n, dim, m, h_init, max_iters, h_map, h_centroids, iters_run))


def kmeans_map(features, m, init, max_iters=100):
    """numpy convenience: (map [n] uint32, centroids [m, dim] float64, assignments made)."""
    F = np.ascontiguousarray(features, dtype=np.float32)
    n, dim = F.shape
    init = np.ascontiguousarray(init, dtype=np.uint32)
    out = np.empty(n, dtype=np.uint32)
    mu = np.empty((m, dim), dtype=np.float64)
    it = ctypes.c_uint32()
    ntc_kmeans_map(F.ctypes.data, n, dim, m, init.ctypes.data, max_iters, out.ctypes.data, mu.ctypes.data,
                   ctypes.byref(it))
    return out, mu, int(it.value)


def ntc_last_error() -> str:
    return _lib.ntc_last_error().decode()


# --------------------------------------------------------- torch convenience

def _ptr(t):
    return None if t is None else t.data_ptr()


def _stream(stream):
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def queries_to_device(q: np.ndarray, device="cuda"):
    """16-byte query records (numpy) -> int32 [n, 4] tensor on the device."""
    import torch
    a = np.ascontiguousarray(q).view(np.int32).reshape(-1, 4)
    return torch.from_numpy(a).to(device)


class Decoder:
    """An ntc context built from an assets object (see ``workloads.Assets``)."""

    def __init__(self, assets, precision: str = "fp16", output: str = "fp32"):
        self._keep = [
            np.ascontiguousarray(assets.level_dims, dtype=np.uint32),
            np.ascontiguousarray(assets.latent_offsets, dtype=np.uint64),
            np.ascontiguousarray(assets.latents, dtype=np.uint16),
            np.ascontiguousarray(assets.weights, dtype=np.float32),
            np.ascontiguousarray(assets.set_to_decoder, dtype=np.uint32),
        ]
        dims, offs, lat, w, m = self._keep
        d = ntc_desc()
        d.num_sets = assets.num_sets
        d.num_decoders = assets.num_decoders
        d.latent_channels = assets.channels
        d.num_levels = assets.num_levels
        d.num_mips = assets.num_mips
        d.level_dims = dims.ctypes.data
        d.latent_offsets = offs.ctypes.data
        d.latents = lat.ctypes.data
        d.num_texels = lat.size // max(1, assets.channels)
        d.in_dim = assets.in_dim
        d.hidden = assets.hidden
        d.num_hidden_layers = assets.num_hidden_layers
        d.out_dim = assets.out_dim
        d.weights = w.ctypes.data
        d.set_to_decoder = m.ctypes.data
        d.precision = PRECISIONS[precision]
        d.address_mode = assets.address_mode
        d.pe_frequencies = getattr(assets, "pe_frequencies", 0)
        d.activation = getattr(assets, "activation", 0)
        d.leaky_slope = getattr(assets, "leaky_slope", 0.0)
        d.output_format = OUTPUTS[output]
        self.desc = d
        self.output = output
        self.out_dim = assets.out_dim
        self.num_decoders = assets.num_decoders
        self.num_levels = assets.num_levels
        self.in_dim = assets.in_dim
        self.ctx = ntc_create(d)
        self._keep = None  # ntc_create copied everything

    def close(self):
        if getattr(self, "ctx", None):
            ntc_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def out_dtype(self):
        import torch
        return torch.float16 if self.output == "fp16" else torch.float32

    def decode(self, queries, out=None, mode: str = "bucketed", stream=None):
        import torch
        n = queries.shape[0]
        if out is None:
            out = torch.empty((n, self.out_dim), dtype=self.out_dtype(), device=queries.device)
        ntc_decode(self.ctx, _ptr(queries), n, _ptr(out), _stream(stream), MODES[mode])
        return out

    def decode_host(self, queries, out=None, mode: str = "bucketed", stream=None):
        import torch
        n = queries.shape[0]
        if out is None:
            out = torch.empty((n, self.out_dim), dtype=self.out_dtype(), pin_memory=True)
        ntc_decode_host(self.ctx, _ptr(queries), n, _ptr(out), _stream(stream), MODES[mode])
        return out

    def taps(self, queries, stream=None):
        import torch
        n = queries.shape[0]
        dev = queries.device
        idx = torch.empty((n, self.num_levels, 2, 4), dtype=torch.int64, device=dev)
        w = torch.empty((n, self.num_levels, 2, 4), dtype=torch.float32, device=dev)
        t = torch.empty((n,), dtype=torch.float32, device=dev)
        ntc_debug_taps(self.ctx, _ptr(queries), n, _ptr(idx), _ptr(w), _ptr(t), _stream(stream))
        return idx, w, t

    def features(self, queries, stream=None):
        import torch
        n = queries.shape[0]
        f = torch.empty((n, self.in_dim), dtype=torch.float32, device=queries.device)
        ntc_debug_features(self.ctx, _ptr(queries), n, _ptr(f), _stream(stream))
        return f

    def decode_rows(self, queries, stream=None):
        """The bucketed tensor-core decode through its debug build: (outputs,
        rows) with rows a numpy structured array of ``DEBUG_ROW`` records
        (ntc_debug_row; rows of bad queries keep their fill of 0xFF bytes)."""
        import torch
        n = queries.shape[0]
        out = torch.empty((n, self.out_dim), dtype=self.out_dtype(), device=queries.device)
        rows = torch.full((max(1, n), DEBUG_ROW.itemsize), 255, dtype=torch.uint8, device=queries.device)
        ntc_debug_decode_rows(self.ctx, _ptr(queries), n, _ptr(out), _ptr(rows), _stream(stream))
        return out, rows[:n].cpu().numpy().view(DEBUG_ROW).reshape(n)

    def bucket(self, queries, stream=None, divergence=False):
        """(perm, counts, tiles) of the bucketing; with divergence=True also
        (copied, sum over 32-query groups of distinct decoders - 1)."""
        import torch
        n = queries.shape[0]
        dev = queries.device
        mt = max(1, ntc_max_tiles(self.ctx, n))
        perm = torch.empty((max(1, n),), dtype=torch.int32, device=dev)
        counts = torch.empty((self.num_decoders + 1,), dtype=torch.int32, device=dev)
        tiles = torch.empty((mt, 3), dtype=torch.int32, device=dev)
        nt = torch.zeros((1,), dtype=torch.int32, device=dev)
        dv = torch.zeros((2,), dtype=torch.int32, device=dev)
        ntc_debug_bucket(self.ctx, _ptr(queries), n, _ptr(perm), _ptr(counts), _ptr(tiles), _ptr(nt), _ptr(dv),
                         _stream(stream))
        k = int(nt.item())
        if divergence:
            c, s = dv.cpu().numpy().astype(np.uint32).tolist()
            return perm[:n], counts, tiles[:k], (c, s)
        return perm[:n], counts, tiles[:k]

    def error_count(self) -> int:
        return ntc_get_error_count(self.ctx)

    def reset_error_count(self):
        ntc_reset_error_count(self.ctx)

    def debug_wait_timeout(self, stream=None):
        """Make one bounded wait give up (a test of the failure path): the next
        error_count() raises NtcError with NTC_ERR_CUDA until reset_error_count()."""
        ntc_debug_wait_timeout(self.ctx, _stream(stream))

    def launches(self) -> int:
        return ntc_launch_count(self.ctx)

    def set_stage_timing(self, enable=True):
        ntc_set_stage_timing(self.ctx, enable)

    def stage_times(self):
        """(bucketing ms, gather-decode ms) of the last decode."""
        return ntc_stage_times(self.ctx)
