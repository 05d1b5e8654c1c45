"""The default tensor-core decode's own addressing and blend, bit for bit.

ntc_debug_decode_rows runs the benchmarked kernel (a debug instantiation of the
same template: same launch configuration, same bucketing) and records every
row its producers build.  Each record is checked against the oracle:
  - the texel index of every tap equals the oracle's (bit-exact);
  - the 16 bytes blended for each tap equal the latents at that index, so the
    row-pair copy and the kernel's own coordinates agree with the oracle's taps;
  - every weight equals the oracle's fp32 bilinear weight times 1 - t (mip lo)
    or t (mip lo + 1), rounded to fp32; in clamp mode an edge row whose two
    texels coincide carries the fp32 sum of both weights on its first tap;
  - the mip pick (lo, t) equals the oracle's;
  - the feature row equals, bit for bit, a numpy replay of the kernel's packed
    fp16 blend from those taps (weights rounded to fp16, each product and
    fused add rounded once, taps in the kernel's order; bf16 rows convert the
    fp16 sums), and lies within a stated bound of the oracle's double-precision
    features (the fp16 blend costs a few fp16 roundings per feature);
  - the outputs equal the production decode's bit for bit.
"""
import functools

import numpy as np
import pytest

import oracle
from paper_2608_27888_gb300 import workloads as W
from tests.util import queries, tiny_assets

pytestmark = pytest.mark.gpu


def ntc():
    from paper_2608_27888_gb300 import ntc as m
    return m


def _bf16_from_f32(x):
    """Round-to-nearest-even fp32 -> bf16 (finite values), as fp32."""
    b = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    b = (b + 0x7FFF + ((b >> 16) & 1)) >> 16
    return (b.astype(np.uint32) << 16).view(np.float32)


def _replay_features(lat16, idx_k, w_k, used, bf16):
    """The kernel's blend of one level for rows with the same tap pattern:
    idx_k [n][slots][4] texel indices, w_k [n][slots][4] fp32 weights, used
    [n][slots] which mip slots the kernel blended.  Returns [n][8] float64."""
    n = idx_k.shape[0]
    acc = None
    for m in range(idx_k.shape[1]):
        for p in range(4):
            x = lat16[idx_k[:, m, p]].astype(np.float64)           # [n][8] fp16 values
            wh = w_k[:, m, p].astype(np.float16).astype(np.float64)[:, None]
            if acc is None:
                acc = (wh * x).astype(np.float16)                     # hmul2: one rounding
            else:
                new = (wh * x + acc.astype(np.float64)).astype(np.float16)  # hfma2: one rounding
                keep = ~used[:, m][:, None]
                acc = np.where(keep, acc, new)
    f = acc.astype(np.float32)
    return (_bf16_from_f32(f) if bf16 else f).astype(np.float64)


def check_rows(a, q, precision):
    m = ntc()
    dec = m.Decoder(a, precision)
    qd = m.queries_to_device(q)
    out_dbg, rows = dec.decode_rows(qd)
    out = dec.decode(qd).cpu().numpy()
    dec.close()
    assert np.array_equal(out_dbg.cpu().numpy().view(np.uint32), out.view(np.uint32)), "outputs differ"
    ri, rw, rt = oracle.taps(a, q)
    good = ri[:, 0, 0, 0] != np.iinfo(np.uint64).max
    assert good.any()
    rows, ri, rw, rt = rows[good], ri[good], rw[good], rt[good]
    n = rows.shape[0]
    two = rt > 0
    # mip pick
    assert np.array_equal(rows["t"].view(np.uint32), rt.view(np.uint32))
    lat16 = a.latents.view(np.float16).reshape(-1, a.channels)
    lat32 = a.latents.view(np.uint32).reshape(-1, a.channels // 2)
    one = np.float32(1.0)
    feats = np.zeros((n, 16))
    for k in range(a.num_levels):
        used = np.stack([np.ones(n, bool), two], axis=1)
        idx = ri[:, k]                                   # [n][2][4]
        w = rw[:, k].copy()
        if a.address_mode == 1:                          # clamp: fold an edge pair's weight
            for r0, r1 in ((0, 1), (2, 3)):
                same = idx[:, :, r0] == idx[:, :, r1]
                w[:, :, r0] = np.where(same, w[:, :, r0] + w[:, :, r1], w[:, :, r0])
                w[:, :, r1] = np.where(same, np.float32(0), w[:, :, r1])
        scale = np.stack([np.where(two, one - rt, one), rt], axis=1).astype(np.float32)  # [n][2]
        w = (w * scale[:, :, None]).astype(np.float32)
        for m_ in range(2):
            sel = used[:, m_]
            assert np.array_equal(rows["idx"][sel, k, m_], idx[sel, m_]), f"level {k} slot {m_} indices"
            assert np.array_equal(rows["w"][sel, k, m_].view(np.uint32), w[sel, m_].view(np.uint32)), \
                f"level {k} slot {m_} weights"
            for p in range(4):
                live = sel & (w[:, m_, p] != 0)
                got = rows["raw"][live, k, m_, p]
                assert np.array_equal(got, lat32[idx[live, m_, p]]), f"level {k} slot {m_} tap {p} bytes"
        feats[:, 8 * k:8 * k + 8] = _replay_features(lat16, idx, w, used, precision == "bf16")
    words = np.ascontiguousarray(rows["feat"]).reshape(n, 8)
    if precision == "fp16":  # feat[i] = inputs 2i (low half) and 2i + 1 (high half)
        got = words.view(np.float16).reshape(n, 16).astype(np.float64)
    else:                    # bf16: a half is the top 16 bits of an fp32
        lo = (words << np.uint32(16)).view(np.float32)
        hi = (words & np.uint32(0xFFFF0000)).view(np.float32)
        got = np.stack([lo, hi], axis=2).reshape(n, 16).astype(np.float64)
    assert np.array_equal(got[:, :8 * a.num_levels], feats[:, :8 * a.num_levels]), "feature rows"
    ref = oracle.features(a, q)[good]
    err = np.abs(got - ref).max()
    # a few fp16 roundings of partial sums bounded by the largest latent
    bound = 12 * 2.0 ** -11 * max(1.0, np.abs(lat16.astype(np.float64)).max())
    if precision == "bf16":
        bound += 2.0 ** -8 * np.abs(ref).max()
    assert err <= bound, f"feature error {err:.3e} above {bound:.3e}"
    return err


@functools.lru_cache(maxsize=None)
def small(name, variant=None):
    return W.named(name, "small", variant)


@pytest.mark.parametrize("name,variant,precision", [
    ("raster-256", None, "fp16"), ("uniform-4m", None, "fp16"), ("gbuffer-1080p", "identity", "fp16"),
    ("gbuffer-1080p", "shared", "fp16"), ("gbuffer-2160p", "128", "fp16"),
    ("gbuffer-2160p-x4-trilinear", None, "fp16"), ("uniform-4m", None, "bf16"),
    ("gbuffer-2160p-x4-trilinear", None, "bf16")])
def test_kernel_rows_on_the_workloads(name, variant, precision):
    w = small(name, variant)
    check_rows(w.assets, w.queries, precision)


@pytest.mark.parametrize("mips", [1, 3])
@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("dims", [(1, 1), (2, 2), (3, 5), (7, 3), (16, 8)])
def test_kernel_rows_on_tiny_grids(mode, dims, mips):
    """Wrap and clamp edges, 1-texel and odd-sized grids, mip blends."""
    W0, H0 = dims
    dims2 = [[(W0, H0), (max(1, W0 // 2), max(1, H0 // 2))]]
    shape = tiny_assets(dims2, num_mips=mips, hidden=64, out_dim=8)
    rng = np.random.default_rng(W0 * 13 + H0 * 5 + mips)
    a = tiny_assets(dims2, num_mips=mips, address_mode=mode, hidden=64, out_dim=8,
                    latents=rng.normal(0.0, 1.0, shape.latents.size),
                    weights=rng.uniform(-0.4, 0.4, shape.weights.shape))
    grid = np.arange(-40, 41) / 16.0
    rows = [(0, float(u), float(v), float(l)) for u in grid[::2] for v in grid[::3]
            for l in (0.0, 0.5, 0.75, 1.25, 2.0, 5.0)]
    rows += [(0, float(u), float(v), float(l)) for u, v, l in
             zip(rng.uniform(-1e3, 1e3, 700), rng.uniform(-3, 3, 700), rng.uniform(-1, 4, 700))]
    check_rows(a, queries(rows), "fp16")
