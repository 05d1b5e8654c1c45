"""GPU parity: libntc (through the C ABI) against the CPU oracle.

Bit-exact: bucketing permutation, counts and tile list; texel indices, bilinear
weights and mip blend factors.  Floating point: fp32 mode within 1e-5 of the
oracle; tensor-core modes within max-abs 2e-2 and mean-abs 2e-3 (outputs are in
[0, 1]).  Small workloads are compared everywhere; full-size workloads in the
launch configuration the benchmark times are compared on sampled queries.
"""
import functools

import numpy as np
import pytest
import torch

import oracle
from paper_2608_27888_gb300 import workloads as W
from tests.util import queries, tiny_assets

pytestmark = pytest.mark.gpu

FP32_TOL = 1e-5
TC_MAX, TC_MEAN = 2e-2, 2e-3
SMALL = [("raster-256", None), ("uniform-4m", None), ("gbuffer-1080p", "identity"),
         ("gbuffer-1080p", "clustered4"), ("gbuffer-1080p", "shared"), ("gbuffer-2160p", "128"),
         ("gbuffer-2160p", "16"), ("gbuffer-2160p", "8"), ("gbuffer-2160p", "1"),
         ("gbuffer-2160p-x4-trilinear", None)]


def ntc():
    from paper_2608_27888_gb300 import ntc as m
    return m


@functools.lru_cache(maxsize=None)
def small(name, variant=None):
    return W.named(name, "small", variant)


@functools.lru_cache(maxsize=None)
def oracle_out(name, variant=None):
    w = small(name, variant)
    return oracle.decode(w.assets, w.queries)


@functools.lru_cache(maxsize=4)
def decoder(name, variant, precision):
    return ntc().Decoder(small(name, variant).assets, precision)


def dq(q):
    return ntc().queries_to_device(q)


def check_tc(got, ref, what):
    err = np.abs(got.astype(np.float64) - ref)
    assert np.isfinite(got).all(), what
    assert err.max() <= TC_MAX, f"{what}: max abs {err.max():.3e}"
    assert err.mean() <= TC_MEAN, f"{what}: mean abs {err.mean():.3e}"


# --------------------------------------------------------------- bucketing

@pytest.mark.parametrize("name,variant", SMALL)
def test_bucketing_bit_exact(name, variant):
    w = small(name, variant)
    dec = decoder(name, variant, "fp16")
    perm, counts, tiles = dec.bucket(dq(w.queries))
    p, c, o, t = oracle.bucket(w.queries["set_id"], w.assets.set_to_decoder, w.assets.num_decoders)
    assert np.array_equal(perm.cpu().numpy().astype(np.uint32), p)
    assert np.array_equal(counts.cpu().numpy().astype(np.uint32), c)
    assert np.array_equal(tiles.cpu().numpy().astype(np.uint32), t)


@pytest.mark.parametrize("n", [1, 31, 32, 33, 127, 128, 129, 4095, 4096, 4097, 70001])
@pytest.mark.parametrize("pattern", ["random", "same", "descending", "bad", "sparse"])
def test_bucketing_edge_cases(n, pattern):
    S, D = 40, 13
    rng = np.random.default_rng(n)
    m = rng.integers(0, D, S).astype(np.uint32)
    m[:3] = [0, 5, 12]
    if pattern == "random":
        sets = rng.integers(0, S, n)
    elif pattern == "same":
        sets = np.full(n, 7)
    elif pattern == "descending":
        sets = (S - 1 - (np.arange(n) * S) // max(n, 1)).clip(0, S - 1)
    elif pattern == "bad":
        sets = rng.integers(0, S + 5, n)  # ids >= S land in the extra bucket
    else:
        sets = rng.choice([1, 2], n)  # most decoders empty
    a = tiny_assets([[(8, 8), (4, 4)]] * S, num_sets=S, num_decoders=D, set_to_decoder=m, hidden=64, out_dim=8)
    q = np.zeros(n, dtype=W.QUERY_DTYPE)
    q["set_id"] = sets
    q["u"] = rng.random(n)
    q["v"] = rng.random(n)
    dec = ntc().Decoder(a, "fp16")
    perm, counts, tiles = dec.bucket(dq(q))
    p, c, o, t = oracle.bucket(q["set_id"], m, D)
    assert np.array_equal(perm.cpu().numpy().astype(np.uint32), p)
    assert np.array_equal(counts.cpu().numpy().astype(np.uint32), c)
    assert np.array_equal(tiles.cpu().numpy().astype(np.uint32), t)
    dec.close()


# ----------------------------------------------------------------- taps

def _taps_equal(dec, a, q):
    idx, wt, t = dec.taps(dq(q))
    ri, rw, rt = oracle.taps(a, q)
    assert np.array_equal(idx.cpu().numpy().view(np.uint64), ri)
    assert np.array_equal(wt.cpu().numpy().view(np.uint32), rw.view(np.uint32))
    assert np.array_equal(t.cpu().numpy().view(np.uint32), rt.view(np.uint32))


@pytest.mark.parametrize("name,variant", [("raster-256", None), ("uniform-4m", None), ("gbuffer-1080p", "identity"),
                                          ("gbuffer-2160p", "128"), ("gbuffer-2160p-x4-trilinear", None)])
def test_taps_bit_exact(name, variant):
    w = small(name, variant)
    _taps_equal(decoder(name, variant, "fp16"), w.assets, w.queries)


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("dims", [(1, 1), (2, 2), (3, 5), (7, 3), (16, 8)])
def test_taps_tiny_grids_bit_exact(mode, dims):
    W0, H0 = dims
    a = tiny_assets([[(W0, H0), (max(1, W0 // 2), max(1, H0 // 2))]], num_mips=3, address_mode=mode,
                    hidden=64, out_dim=8)
    grid = np.arange(-40, 41) / 16.0
    rng = np.random.default_rng(W0 * 7 + H0)
    rows = [(0, float(u), float(v), float(l)) for u in grid[::3] for v in grid[::4]
            for l in (0.0, 0.5, 1.25, 2.0, 5.0)]
    rows += [(0, float(u), float(v), float(l)) for u, v, l in
             zip(rng.uniform(-1e3, 1e3, 500), rng.uniform(-3, 3, 500), rng.uniform(-1, 4, 500))]
    dec = ntc().Decoder(a, "fp32")
    _taps_equal(dec, a, queries(rows))
    dec.close()


@pytest.mark.parametrize("mips", [1, 3])
@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("dims", [(1, 1), (2, 2), (3, 5), (7, 3), (16, 8)])
def test_decode_tc_tiny_grids_edges(mode, dims, mips):
    """The tensor-core path reads each bilinear row as a texel pair: wrap and
    clamp edges, 1-texel grids and mip blends must still match the oracle."""
    W0, H0 = dims
    dims2 = [[(W0, H0), (max(1, W0 // 2), max(1, H0 // 2))]]
    shape = tiny_assets(dims2, num_mips=mips, hidden=64, out_dim=8)
    rng = np.random.default_rng(W0 * 31 + H0 * 7 + mips)
    a = tiny_assets(dims2, num_mips=mips, address_mode=mode, hidden=64, out_dim=8,
                    latents=rng.normal(0.0, 1.0, shape.latents.size),
                    weights=rng.uniform(-0.4, 0.4, shape.weights.shape))
    grid = np.arange(-40, 41) / 16.0
    rows = [(0, float(u), float(v), float(l)) for u in grid for v in grid[::2] for l in (0.0, 0.75, 2.0)]
    q = queries(rows)
    ref, _ = oracle.decode(a, q)
    for prec in ("fp16", "bf16"):
        dec = ntc().Decoder(a, prec)
        check_tc(dec.decode(dq(q)).cpu().numpy(), ref, f"{dims} mode {mode} mips {mips} {prec}")
        dec.close()


@pytest.mark.parametrize("name,variant", [("uniform-4m", None), ("gbuffer-2160p-x4-trilinear", None)])
def test_features_match_oracle(name, variant):
    w = small(name, variant)
    f = decoder(name, variant, "fp16").features(dq(w.queries)).cpu().numpy()
    ref = oracle.features(w.assets, w.queries)
    assert np.abs(f - ref).max() <= 1e-5 * max(1.0, np.abs(ref).max())


# --------------------------------------------------------------- decode

@pytest.mark.parametrize("mode", ["bucketed", "divergent_fma"])
@pytest.mark.parametrize("name,variant", SMALL)
def test_decode_fp32_mode(name, variant, mode):
    w = small(name, variant)
    ref, _ = oracle_out(name, variant)
    got = decoder(name, variant, "fp32").decode(dq(w.queries), mode=mode).cpu().numpy()
    assert np.abs(got - ref).max() <= FP32_TOL


@pytest.mark.parametrize("precision", ["fp16", "bf16"])
@pytest.mark.parametrize("mode", ["bucketed", "bucketed_mma", "divergent", "divergent_fma"])
@pytest.mark.parametrize("name,variant", SMALL)
def test_decode_tensor_core_modes(name, variant, mode, precision):
    w = small(name, variant)
    ref, _ = oracle_out(name, variant)
    got = decoder(name, variant, precision).decode(dq(w.queries), mode=mode).cpu().numpy()
    check_tc(got, ref, f"{name}/{variant} {mode} {precision}")


def test_hidden_128_and_9_channels_on_all_paths():
    w = small("gbuffer-2160p-x4-trilinear")
    ref, _ = oracle_out("gbuffer-2160p-x4-trilinear")
    for prec, modes in (("fp32", ["bucketed", "divergent_fma"]),
                        ("fp16", ["bucketed", "bucketed_mma", "divergent", "divergent_fma"]),
                        ("bf16", ["divergent_fma"])):
        dec = decoder("gbuffer-2160p-x4-trilinear", None, prec)
        for m in modes:
            got = dec.decode(dq(w.queries), mode=m).cpu().numpy()
            if prec == "fp32":
                assert np.abs(got - ref).max() <= FP32_TOL
            else:
                check_tc(got, ref, m)


@pytest.mark.parametrize("mode", ["bucketed", "bucketed_mma", "divergent", "divergent_fma"])
def test_order_invariance_is_bitwise(mode):
    w = small("gbuffer-1080p", "clustered4")
    dec = decoder("gbuffer-1080p", "clustered4", "fp16")
    out = dec.decode(dq(w.queries), mode=mode).cpu().numpy()
    p = np.random.default_rng(1).permutation(len(w.queries))
    out2 = dec.decode(dq(w.queries[p]), mode=mode).cpu().numpy()
    # every row's arithmetic is independent of the other rows of its tile or
    # warp (the divergent kernels mask, they do not mix rows)
    assert np.array_equal(out2, out[p])


def test_bad_queries_nan_and_counted():
    w = small("uniform-4m")
    q = w.queries[:5000].copy()
    q["set_id"][::97] = 999
    q["u"][5::101] = np.nan
    q["v"][7::103] = np.inf
    nbad = len(set(range(0, 5000, 97)) | set(range(5, 5000, 101)) | set(range(7, 5000, 103)))
    ref, bad = oracle.decode(w.assets, q)
    assert bad == nbad
    for prec, mode in (("fp32", "bucketed"), ("fp16", "bucketed"), ("fp16", "bucketed_mma"),
                       ("fp16", "divergent"), ("fp16", "divergent_fma"), ("fp32", "divergent_fma")):
        dec = ntc().Decoder(w.assets, prec)
        got = dec.decode(dq(q), mode=mode).cpu().numpy()
        assert np.array_equal(np.isnan(got), np.isnan(ref)), (prec, mode)
        assert dec.error_count() == nbad, (prec, mode)
        dec.reset_error_count()
        assert dec.error_count() == 0
        dec.close()


@pytest.mark.parametrize("precision,output", [("fp16", "fp32"), ("bf16", "fp32"), ("fp16", "fp16")])
def test_tiles_of_bad_queries_at_hidden_128(precision, output):
    """40 % of the queries have out-of-range set ids: their bucket (the last)
    is about 200 tiles with nothing to multiply, so the issuer warps of the
    H = 128 kernel hand over runs of such tiles back to back."""
    w = small("gbuffer-2160p-x4-trilinear")
    q = w.queries.copy()
    i = np.arange(len(q))
    q["set_id"][i % 5 < 2] = 1000 + (i[i % 5 < 2] % 7)
    q["u"][3::211] = np.nan
    ref, nbad = oracle.decode(w.assets, q)
    assert nbad > 0.4 * len(q)
    dec = ntc().Decoder(w.assets, precision, output=output)
    got = dec.decode(dq(q)).float().cpu().numpy()
    bad = np.isnan(ref).any(axis=1)
    assert np.array_equal(np.isnan(got).any(axis=1), bad)
    assert np.isnan(got[bad]).all()
    check_tc(got[~bad], ref[~bad], f"{precision}/{output}")
    assert dec.error_count() == nbad
    dec.close()


def test_decode_host_equals_device_decode():
    w = small("gbuffer-1080p", "identity")
    dec = decoder("gbuffer-1080p", "identity", "fp16")
    dev = dec.decode(dq(w.queries)).cpu().numpy()
    hq = torch.from_numpy(np.ascontiguousarray(w.queries).view(np.int32).reshape(-1, 4)).pin_memory()
    host = dec.decode_host(hq).numpy()
    assert np.array_equal(host, dev)


@pytest.mark.parametrize("output", ["fp32", "fp16"])
@pytest.mark.parametrize("n", [3 * 2 ** 18 + 777, 4 * 2 ** 20 - 5, 4 * 2 ** 20])
def test_decode_host_over_many_chunks(n, output):
    """ntc_decode_host pipelines chunks of at least 2^18 queries (up to 32 of
    them), each bucketed on its own.  On a fully divergent stream (every chunk
    copies its records) the rows must equal one device-buffer decode over all
    n bit for bit, with the last chunk ragged or full."""
    w = W.named("uniform-4m", "full")
    q = w.queries[:n]
    dec = ntc().Decoder(w.assets, "fp16", output=output)
    dev = dec.decode(dq(q)).cpu()
    hq = torch.from_numpy(np.ascontiguousarray(q).view(np.int32).reshape(-1, 4)).pin_memory()
    host = dec.decode_host(hq)
    bits = torch.int16 if output == "fp16" else torch.int32
    assert torch.equal(host.view(bits), dev.view(bits))
    # a second call reuses the staging and the events
    host2 = dec.decode_host(hq)
    assert torch.equal(host2.view(bits), dev.view(bits))
    # pageable buffers: the copies no longer overlap, the rows are the same
    pq = torch.empty(hq.shape, dtype=hq.dtype)
    pq.copy_(hq)
    pout = torch.empty(dev.shape, dtype=dev.dtype)
    dec.decode_host(pq, pout)
    assert torch.equal(pout.view(bits), dev.view(bits))
    dec.close()


NO_PDL_CASES = [("gbuffer-2160p-x4-trilinear", None), ("uniform-4m", None), ("gbuffer-1080p", "clustered4"),
                ("gbuffer-1080p", "shared")]


def test_ordinary_launches_give_the_same_rows(tmp_path):
    """With NTC_NO_PDL set the bucketing and decode kernels are ordinary
    launches instead of programmatic dependents; a process decoding that way
    must produce the same bits, through device and host buffers."""
    import os
    import subprocess
    import sys
    import textwrap
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    script = textwrap.dedent(f"""
        import sys
        import numpy as np
        import torch
        sys.path.insert(0, {root!r})
        from paper_2608_27888_gb300 import ntc, workloads as W
        for i, (name, variant) in enumerate({NO_PDL_CASES!r}):
            w = W.named(name, "small", variant)
            dec = ntc.Decoder(w.assets, "fp16")
            np.save({str(tmp_path)!r} + f"/dev{{i}}.npy", dec.decode(ntc.queries_to_device(w.queries)).cpu().numpy())
            hq = torch.from_numpy(np.ascontiguousarray(w.queries).view(np.int32).reshape(-1, 4)).pin_memory()
            np.save({str(tmp_path)!r} + f"/host{{i}}.npy", dec.decode_host(hq).numpy())
            dec.close()
    """)
    env = dict(os.environ, NTC_NO_PDL="1")
    r = subprocess.run([sys.executable, "-c", script], env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    for i, (name, variant) in enumerate(NO_PDL_CASES):
        w = small(name, variant)
        dec = ntc().Decoder(w.assets, "fp16")
        got = dec.decode(dq(w.queries)).cpu().numpy()
        dec.close()
        for kind in ("dev", "host"):
            other = np.load(tmp_path / f"{kind}{i}.npy")
            assert np.array_equal(got.view(np.uint32), other.view(np.uint32)), (name, variant, kind)


def test_empty_and_invalid_calls():
    m = ntc()
    dec = decoder("raster-256", None, "fp16")
    empty = torch.empty((0, 4), dtype=torch.int32, device="cuda")
    out = dec.decode(empty)
    assert out.shape == (0, 8)
    with pytest.raises(m.NtcError):
        m.ntc_decode(dec.ctx, 0, 10, 0, 0, m.NTC_MODE_BUCKETED)
    with pytest.raises(m.NtcError):
        fp32 = decoder("raster-256", None, "fp32")
        fp32.decode(dq(small("raster-256").queries[:64]), mode="divergent")


# ------------------------------------------------- full sizes, sampled check

FULL = [("raster-256", None), ("uniform-4m", None), ("gbuffer-1080p", "identity"), ("gbuffer-2160p", "128"),
        ("gbuffer-2160p-x4-trilinear", None)]


@pytest.mark.parametrize("name,variant", FULL)
def test_full_size_sampled(name, variant):
    w = W.named(name, "full", variant)
    n = len(w.queries)
    rng = np.random.default_rng(W.WORKLOADS.index(name) + 1)
    sample = np.unique(np.concatenate([rng.integers(0, n, 20000), np.arange(min(n, 4096)),
                                       np.arange(max(0, n - 300), n)]))
    ref, _ = oracle.decode(w.assets, w.queries[sample])
    qd = dq(w.queries)
    dec = ntc().Decoder(w.assets, "fp16")
    out = dec.decode(qd, mode="bucketed")
    got = out[torch.from_numpy(sample).cuda()].cpu().numpy()
    check_tc(got, ref, f"{w.name} bucketed")
    for mode in ("divergent", "divergent_fma"):
        div = dec.decode(qd, mode=mode)[torch.from_numpy(sample).cuda()].cpu().numpy()
        check_tc(div, ref, f"{w.name} {mode}")
    perm, counts, tiles = dec.bucket(qd)
    p, c, _, t = oracle.bucket(w.queries["set_id"], w.assets.set_to_decoder, w.assets.num_decoders)
    assert np.array_equal(perm.cpu().numpy().astype(np.uint32), p)
    assert np.array_equal(counts.cpu().numpy().astype(np.uint32), c)
    assert np.array_equal(tiles.cpu().numpy().astype(np.uint32), t)
    idx, wt, tt = dec.taps(dq(w.queries[sample]))
    ri, rw, rt = oracle.taps(w.assets, w.queries[sample])
    assert np.array_equal(idx.cpu().numpy().view(np.uint64), ri)
    assert np.array_equal(wt.cpu().numpy().view(np.uint32), rw.view(np.uint32))
    dec.close()
    del out, qd
    torch.cuda.empty_cache()


# ------------------------------------------ single-decoder and mixed warps

def _coherent_case(kind, n, rng, assets, base):
    """Query streams of engineered warps: warps whose sets differ but share one
    decoder, one bad set id inside an otherwise single-decoder warp, warps
    alternating between one decoder and uniform sets, ragged tails."""
    q = base[:n].copy()
    S = assets.num_sets
    m = assets.set_to_decoder
    by_dec = {d: np.flatnonzero(m == d) for d in range(assets.num_decoders)}
    nw = (n + 31) // 32
    sets = np.empty(nw * 32, dtype=np.uint32)
    for w in range(nw):
        d = rng.integers(0, assets.num_decoders)
        if kind == "coherent":
            sets[32 * w:32 * w + 32] = rng.choice(by_dec[d], 32)  # one decoder, several sets
        elif kind == "alternating":
            sets[32 * w:32 * w + 32] = rng.choice(by_dec[d], 32) if w % 2 else rng.integers(0, S, 32)
        elif kind == "bad_inside":
            sets[32 * w:32 * w + 32] = rng.choice(by_dec[d], 32)
            if w % 3 == 0:
                sets[32 * w + rng.integers(0, 32)] = S + 5  # out of range: the warp is mixed
        else:
            raise ValueError(kind)
    q["set_id"] = sets[:n]
    return q


@pytest.mark.parametrize("variant", ["clustered4", "shared"])
@pytest.mark.parametrize("kind", ["coherent", "alternating", "bad_inside"])
@pytest.mark.parametrize("n", [1, 31, 32, 33, 127, 129, 2047, 2048, 2081, 20000 + 17])
def test_single_decoder_and_mixed_warps(kind, n, variant):
    """With one shared decoder ("shared") the tensor-core path sorts nothing and
    decodes the queries in their own order; with four it buckets them."""
    base_w = small("gbuffer-1080p", variant)
    a = base_w.assets
    rng = np.random.default_rng(n * 7 + len(kind))
    base = np.resize(base_w.queries, max(n, 1))
    q = _coherent_case(kind, n, rng, a, base)
    ref, nbad = oracle.decode(a, q)
    dec = decoder("gbuffer-1080p", variant, "fp16")
    dec.reset_error_count()
    got = dec.decode(dq(q), mode="bucketed").cpu().numpy()
    assert np.array_equal(np.isnan(got), np.isnan(ref))
    ok = ~np.isnan(ref).any(1)
    check_tc(got[ok], ref[ok], f"coherent {kind} n={n}")
    assert dec.error_count() == nbad
    # a permutation scatters the single-decoder warps into mixed ones: every
    # row must come out bit for bit the same either way
    p = rng.permutation(n)
    got_p = dec.decode(dq(q[p]), mode="bucketed").cpu().numpy()
    assert np.array_equal(got_p[ok[p]], got[p][ok[p]])
    dec.reset_error_count()


# ------------------------------------------------- k-means map source (Alg. 2)

def _km_case(case):
    rng = np.random.default_rng(len(case))
    if case == "categories":  # the 586 synthetic 512-d embeddings, 11 groups
        F = W.embeddings(W.BASE_SEED, W.CATEGORY_SIZES)
        return F, 11, W.kmeans_init(W.BASE_SEED, len(F), 11), 100
    if case == "many_groups":
        F = rng.standard_normal((2000, 24)).astype(np.float32)
        return F, 70, rng.permutation(2000)[:70], 200
    if case == "single":
        F = rng.standard_normal((33, 7)).astype(np.float32)
        return F, 1, [5], 10
    if case == "every_row":
        F = rng.standard_normal((50, 3)).astype(np.float32)
        return F, 50, rng.permutation(50), 10
    if case == "dim1_ties":  # repeated values: exact distance ties
        F = rng.integers(0, 4, (300, 1)).astype(np.float32)
        return F, 3, [0, 1, 2] if len(set(F[:3, 0])) == 3 else rng.permutation(300)[:3], 50
    if case == "one_iteration":
        F = rng.standard_normal((400, 16)).astype(np.float32)
        return F, 8, rng.permutation(400)[:8], 1
    raise ValueError(case)


@pytest.mark.parametrize("case", ["categories", "many_groups", "single", "every_row", "dim1_ties",
                                  "one_iteration"])
def test_kmeans_map_equals_oracle_bit_for_bit(case):
    F, m, init, iters = _km_case(case)
    init = np.asarray(init, dtype=np.uint32)
    if len(set(init.tolist())) < m:
        pytest.skip("start rows not distinct")
    ref_map, ref_mu, ref_it = oracle.kmeans(F, m, init, max_iters=iters)
    got_map, got_mu, got_it = ntc().kmeans_map(F, m, init, max_iters=iters)
    assert got_it == ref_it
    assert np.array_equal(got_map, ref_map)
    assert np.array_equal(got_mu.view(np.uint64), ref_mu.view(np.uint64))


def test_bucketing_with_the_most_decoders():
    """4095 decoders (the most the library accepts): the bucketing kernels'
    per-warp counters then take most of their shared memory."""
    D = 4095
    a = tiny_assets([[(4, 4), (2, 2)]] * D, hidden=16, out_dim=4, num_decoders=D, num_sets=D,
                    set_to_decoder=np.random.default_rng(0).permutation(D))
    dec = ntc().Decoder(a, "fp16")
    rng = np.random.default_rng(1)
    for n in (1, 2049, 70001):
        sets = rng.integers(0, D + 3, n)  # a few out-of-range ids: the extra bucket
        q = queries([(int(s), 0.5, 0.5, 0.0) for s in sets])
        perm, counts, tiles = dec.bucket(dq(q))
        p, c, _, t = oracle.bucket(q["set_id"], a.set_to_decoder, D)
        assert np.array_equal(perm.cpu().numpy().astype(np.uint32), p)
        assert np.array_equal(counts.cpu().numpy().astype(np.uint32), c)
        assert np.array_equal(tiles.cpu().numpy().astype(np.uint32), t)
    dec.close()


@pytest.mark.parametrize("pattern", ["random", "same", "bad", "sparse"])
def test_bucketed_decode_writes_every_row(pattern):
    """The tensor-core decode sorts with the three-kernel counting sort
    (per-chunk counts, a scan whose last CTA clears the ticket, stable
    placement).  Every row of the output must be written exactly as the
    oracle decodes it, over chunk boundaries and ragged tails, on consecutive
    calls of varying sizes."""
    S, D = 40, 13
    rng = np.random.default_rng(7)
    m = rng.integers(0, D, S).astype(np.uint32)
    a = tiny_assets([[(8, 8), (4, 4)]] * S, num_sets=S, num_decoders=D, set_to_decoder=m, hidden=64, out_dim=8)
    dec = ntc().Decoder(a, "fp16")
    for n in (1, 2047, 2048, 2049, 3 * 2048 + 77, 70001, 129):
        if pattern == "random":
            sets = rng.integers(0, S, n)
        elif pattern == "same":
            sets = np.full(n, 7)
        elif pattern == "bad":
            sets = rng.integers(0, S + 5, n)
        else:
            sets = rng.choice([1, 2], n)
        q = np.zeros(n, dtype=W.QUERY_DTYPE)
        q["set_id"] = sets
        q["u"] = rng.random(n)
        q["v"] = rng.random(n)
        ref, nbad = oracle.decode(a, q)
        out = torch.full((n, 8), -7.0, device="cuda")
        dec.reset_error_count()
        got = dec.decode(dq(q), out=out).cpu().numpy()
        assert not (got == -7.0).any(), n
        bad = np.isnan(ref).any(1)
        assert np.array_equal(np.isnan(got).any(1), bad), n
        if (~bad).any():
            check_tc(got[~bad], ref[~bad], f"n={n}")
        assert dec.error_count() == nbad
    dec.close()


def test_a_wait_that_gives_up_is_reported_and_the_context_recovers():
    """Every mbarrier wait is bounded (200 ms).  A wait that gives up records
    it in the context's status word: error_count() then fails with
    NTC_ERR_CUDA until the reset, and the context decodes correctly after."""
    m = ntc()
    w = small("uniform-4m")
    dec = decoder("uniform-4m", None, "fp16")
    dec.reset_error_count()
    dec.debug_wait_timeout()
    with pytest.raises(m.NtcError) as e:
        dec.error_count()
    assert e.value.status == m.NTC_ERR_CUDA
    dec.reset_error_count()
    assert dec.error_count() == 0
    got = dec.decode(dq(w.queries)).cpu().numpy()
    ref, _ = oracle_out("uniform-4m")
    check_tc(got, ref, "after a wait gave up")


@pytest.mark.parametrize("hidden,out_dim,mips", [(64, 8, 1), (128, 9, 2)])
def test_every_tile_switches_decoder(hidden, out_dim, mips):
    """The most decoder changes the tensor-core decode can meet: 4095 decoders
    of exactly 8 tiles (1024 queries) each, so the next tile of every consumer
    (4 x 152 tiles later at H = 64, 2 x 152 at H = 128) belongs to another
    decoder and the weight image is reloaded before every tile.  The reload must
    wait for the previous tile's output layer, which still reads W3 of the
    image (Sec. 3.3: every row is decoded by its own decoder D_c(i)).  Every row
    is compared with the oracle."""
    D, per = 4095, 1024
    seed = W.BASE_SEED + 900 + hidden
    a = W.make_assets(seed, D, 16, mips, D, W.map_identity(D), hidden=hidden, out_dim=out_dim)
    n = D * per
    rng = np.random.default_rng(seed)
    q = np.zeros(n, dtype=W.QUERY_DTYPE)
    q["set_id"] = rng.permutation(np.repeat(np.arange(D, dtype=np.uint32), per))
    q["u"] = rng.random(n, dtype=np.float32)
    q["v"] = rng.random(n, dtype=np.float32)
    q["lod"] = rng.random(n, dtype=np.float32) if mips > 1 else 0.0
    ref, _ = oracle.decode(a, q)
    dec = ntc().Decoder(a, "fp16")
    for _ in range(2):
        got = dec.decode(dq(q)).cpu().numpy()
        check_tc(got, ref, f"H={hidden} every tile a new decoder")
    assert dec.error_count() == 0
    dec.close()
    torch.cuda.empty_cache()


# ------------------------------- divergence-aware bucketing (Sec. 2, Eq. 1)

def _eq1_sum(q, a):
    ids = oracle.decoder_ids(q["set_id"], a.set_to_decoder, a.num_decoders)
    return int((oracle.divergence_map(ids, 32) - 1).sum())


@pytest.mark.parametrize("name,variant", SMALL)
def test_divergence_score_and_copy_decision_match_the_oracle(name, variant):
    """k_count sums Eq. 1's |D_w - 1| over the 32-query groups; the records are
    copied in bucket order exactly when that mean exceeds 4."""
    w = small(name, variant)
    if w.assets.num_decoders == 1 and name != "uniform-4m":
        pytest.skip("one decoder: nothing is bucketed")
    _, _, _, (copied, s) = decoder(name, variant, "fp16").bucket(dq(w.queries), divergence=True)
    ref = _eq1_sum(w.queries, w.assets)
    groups = (len(w.queries) + 31) // 32
    assert s == ref
    assert copied == int(ref > 4 * groups)


@pytest.mark.parametrize("d", [1, 2, 4, 5, 6, 8, 16, 32])
def test_divergence_sweep_decodes_on_both_sides_of_the_copy_threshold(d):
    """Exactly d distinct decoders in every warp: d <= 5 reads the queries
    through perm, d >= 6 reads copied records (Eq. 1 score d - 1 against 4).
    Outputs are compared with the oracle, the perm with its stable sort."""
    wl = W.sweep(d, 256, "small")
    a, q = wl.assets, wl.queries
    dec = ntc().Decoder(a, "fp16")
    perm, _, _, (copied, s) = dec.bucket(dq(q), divergence=True)
    groups = (len(q) + 31) // 32
    assert s == _eq1_sum(q, a) == (d - 1) * groups
    assert copied == int(d - 1 > 4)
    p, _, _, _ = oracle.bucket(q["set_id"], a.set_to_decoder, a.num_decoders)
    assert np.array_equal(perm.cpu().numpy().astype(np.uint32), p)
    ref, _ = oracle.decode(a, q)
    for prec in ("fp16", "bf16"):
        d2 = dec if prec == "fp16" else ntc().Decoder(a, prec)
        check_tc(d2.decode(dq(q)).cpu().numpy(), ref, f"sweep d={d} {prec}")
        if d2 is not dec:
            d2.close()
    fp = ntc().Decoder(a, "fp32")
    assert np.abs(fp.decode(dq(q)).cpu().numpy() - ref).max() <= FP32_TOL
    assert np.abs(dec.decode(dq(q), mode="bucketed_mma").cpu().numpy() - ref).max() <= TC_MAX
    fp.close()
    dec.close()
