"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: hand-derived
taps, closed forms (texel centres, constant and linear grids, zero and identity
MLPs), a library routine (torch.nn.functional.linear in fp64), brute force on
tiny inputs, and the numbers printed in the paper (Tables 1, 5, 6; Eq. 1).
"""
import json
import os
import random

import numpy as np
import pytest
import torch

import oracle
from paper_2608_27888_gb300 import workloads as W
from tests.util import queries, split_weights, tiny_assets

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def sigmoid(x):
    return 1.0 / (1.0 + np.exp(-x))


# ------------------------------------------------------------------ taps (a3)

def _single_level(W0, H0, mips, mode, latents=None):
    return tiny_assets([[(W0, H0)]], num_mips=mips, address_mode=mode, latents=latents)


def test_taps_hand_derived():
    cases = json.load(open(os.path.join(GOLD, "taps_handworked.json")))["cases"]
    for c in cases:
        a = _single_level(c["W0"], c["H0"], c["mips"], {"wrap": 0, "clamp": 1}[c["mode"]])
        idx, w, t = oracle.taps(a, queries([(0, c["u"], c["v"], c["lod"])]))
        assert idx[0, 0, 0].tolist() == c["lo"], c["why"]
        assert w[0, 0, 0].tolist() == c["w_lo"], c["why"]
        assert float(t[0]) == c["t"], c["why"]
        if "hi" in c:
            assert idx[0, 0, 1].tolist() == c["hi"], c["why"]
            assert w[0, 0, 1].tolist() == c["w_hi"], c["why"]
        else:
            assert (idx[0, 0, 1] == np.uint64(2**64 - 1)).all()
            assert (w[0, 0, 1] == 0).all()


@pytest.mark.parametrize("W0,H0", [(1, 1), (2, 2), (3, 5), (8, 4), (16, 16)])
@pytest.mark.parametrize("mode", [0, 1])
def test_texel_centres_return_grid_values_exactly(W0, H0, mode):
    rng = np.random.default_rng(W0 * 100 + H0)
    vals = rng.standard_normal((H0, W0, 8)).astype(np.float16)
    a = _single_level(W0, H0, 1, mode, latents=vals.astype(np.float32))
    rows = []
    for j in range(H0):
        for i in range(W0):
            rows.append((0, (i + 0.5) / W0, (j + 0.5) / H0, 0.0))
    f = oracle.features(a, queries(rows))
    assert np.array_equal(f, vals.reshape(-1, 8).astype(np.float64))
    idx, w, _ = oracle.taps(a, queries(rows))
    assert (w[:, 0, 0, 0] == 1.0).all() and (w[:, 0, 0, 1:] == 0.0).all()


def test_wrap_is_periodic_and_weights_partition_unity():
    a = _single_level(8, 4, 1, 0)
    grid = np.arange(-64, 64) / 16.0  # dyadic UVs, negative and above 1
    rows = [(0, u, v, 0.0) for u in grid[::3] for v in grid[::5]]
    q = queries(rows)
    idx, w, _ = oracle.taps(a, q)
    q2 = q.copy()
    q2["u"] += 3.0
    q2["v"] -= 2.0
    idx2, w2, _ = oracle.taps(a, q2)
    assert np.array_equal(idx, idx2) and np.array_equal(w, w2)
    assert np.all(w[:, 0, 0].astype(np.float64).sum(-1) == 1.0)


def test_linear_ramp_interpolates_linearly():
    # L[j][i][c] = (c + 1) * i - 0.5 * c * j: exact in fp16, linear in (i, j), so
    # bilinear interpolation away from the wrap seam is the same linear function
    # of the continuous coordinates x = u W - 0.5, y = v H - 0.5 (channel order
    # and axis roles both matter here).
    W0, H0 = 16, 8
    j, i, c = np.meshgrid(np.arange(H0), np.arange(W0), np.arange(8), indexing="ij")
    lat = ((c + 1) * i - 0.5 * c * j).astype(np.float32)
    a = _single_level(W0, H0, 1, 0, latents=lat)
    us = (np.arange(1, 30) / 32.0 + 0.5 / W0)
    vs = (np.arange(1, 14) / 16.0 + 0.5 / H0)
    rows = [(0, u, v, 0.0) for u in us for v in vs if u * W0 - 0.5 <= W0 - 1 and v * H0 - 0.5 <= H0 - 1]
    q = queries(rows)
    f = oracle.features(a, q)
    x = q["u"].astype(np.float64) * W0 - 0.5
    y = q["v"].astype(np.float64) * H0 - 0.5
    ch = np.arange(8)
    expect = (ch[None] + 1) * x[:, None] - 0.5 * ch[None] * y[:, None]
    assert np.allclose(f, expect, atol=1e-12, rtol=0)


# ------------------------------------------------------------- features (a4)

def test_constant_grid_gives_constant_features_at_every_mip_and_blend():
    dims = [[(16, 8), (8, 4)]]
    Wd, offs, total = W.pyramid_layout(1, dims, 3)
    lat = np.zeros((total, 8), dtype=np.float32)
    lat[:] = np.array([0.5, -1.25, 2.0, 0.0, 3.5, -0.75, 1.0, 0.125])
    a = tiny_assets(dims, num_mips=3, latents=lat)
    rng = np.random.default_rng(7)
    rows = [(0, float(u), float(v), float(l)) for u, v, l in
            zip(rng.uniform(-3, 3, 300), rng.uniform(-3, 3, 300), rng.uniform(-1, 4, 300))]
    f = oracle.features(a, queries(rows))
    expect = np.concatenate([lat[0], lat[0]])
    # the four fp32 tap weights sum to 1 up to their own rounding (a few 2^-24)
    assert np.allclose(f, expect[None], atol=4 * 2.0**-24 * 3.5, rtol=0)


def test_levels_concatenate_in_order():
    dims = [[(4, 4), (2, 2)]]
    _, offs, total = W.pyramid_layout(1, dims, 1)
    lat = np.zeros((total, 8), dtype=np.float32)
    lat[:16] = 1.5    # level 0
    lat[16:] = -2.25  # level 1
    a = tiny_assets(dims, num_mips=1, latents=lat)
    f = oracle.features(a, queries([(0, 0.3, 0.7, 0.0), (0, -5.1, 9.3, 0.0)]))
    assert np.allclose(f, np.array([[1.5] * 8 + [-2.25] * 8] * 2), atol=4 * 2.0**-24 * 2.25, rtol=0)


def test_trilinear_blend_of_constant_mips():
    # mip m of the single level is filled with the constant c_m, so the feature
    # is (1 - t) c_lo + t c_hi with lo = floor(lod), t = lod - lo (lod clamped
    # to [0, last mip]).
    cm = [1.0, -2.0, 4.0]
    dims = [[(8, 8)]]
    _, offs, total = W.pyramid_layout(1, dims, 3)
    lat = np.zeros((total, 8), dtype=np.float32)
    for m in range(3):
        start = int(offs[0, 0, m])
        end = int(offs[0, 0, m + 1]) if m < 2 else total
        lat[start:end] = cm[m]
    a = tiny_assets(dims, num_mips=3, latents=lat)
    lods = [0.0, 0.25, 0.5, 1.0, 1.75, 2.0, 2.5, 9.0, -1.0]
    f = oracle.features(a, queries([(0, 0.37, 0.61, l) for l in lods]))
    for l, row in zip(lods, f):
        lam = min(max(l, 0.0), 2.0)
        lo = int(np.floor(lam))
        t = lam - lo
        hi = min(lo + 1, 2)
        assert np.allclose(row, (1 - t) * cm[lo] + t * cm[hi], atol=4 * 2.0**-24 * 4)


def test_fractional_lod_blends_the_two_integral_lods():
    # with t = 0 only mip lo is read; with t > 0 the feature is the linear blend
    # of the features the same UV gets at lod = lo and lod = lo + 1.
    w = W.named("gbuffer-2160p-x4-trilinear", "small")
    q = w.queries[:3000].copy()
    lo = np.floor(q["lod"])
    t = (q["lod"] - lo).astype(np.float64)
    qa, qb = q.copy(), q.copy()
    qa["lod"], qb["lod"] = lo, lo + 1
    f, fa, fb = (oracle.features(w.assets, x) for x in (q, qa, qb))
    assert np.allclose(f, (1 - t)[:, None] * fa + t[:, None] * fb, atol=1e-12)
    _, wt, tt = oracle.taps(w.assets, qa)
    assert (tt == 0).all() and (wt[:, :, 1] == 0).all()


# -------------------------------------------------------------------- MLP

def _random_assets(seed, hidden=16, out_dim=5, layers=2, num_decoders=1, num_sets=1, mode=0):
    rng = np.random.default_rng(seed)
    dims = [[(8, 8), (4, 4)]] * num_sets
    _, _, total = W.pyramid_layout(num_sets, dims, 2)
    lat = rng.standard_normal(total * 8).astype(np.float32) * 0.5
    a = tiny_assets(dims, num_mips=2, latents=lat, hidden=hidden, out_dim=out_dim, layers=layers,
                    num_decoders=num_decoders, num_sets=num_sets,
                    set_to_decoder=rng.integers(0, num_decoders, num_sets), address_mode=mode)
    a.weights[:] = rng.uniform(-0.6, 0.6, a.weights.shape).astype(np.float32)
    return a, rng


def test_zero_weights_give_sigmoid_of_output_bias():
    a, rng = _random_assets(1)
    a.weights[:] = 0
    Ws = split_weights(a)
    Ws[-1][:] = np.array([0.5, -1.0, 2.0, 0.0, -3.0], dtype=np.float32)
    Ws[1][:] = 1.0  # hidden biases must not leak through zero output weights
    q = queries([(0, float(u), float(v), 0.3) for u, v in rng.uniform(-2, 2, (50, 2))])
    out, bad = oracle.decode(a, q)
    assert bad == 0
    assert np.allclose(out, sigmoid(np.array([0.5, -1.0, 2.0, 0.0, -3.0]))[None], atol=1e-15)


def test_identity_weights_give_sigmoid_of_relu_features():
    a, rng = _random_assets(2, hidden=16, out_dim=8)
    a.weights[:] = 0
    W1, b1, W2, b2, W3, b3 = split_weights(a)
    W1[:] = np.eye(16)
    W2[:] = np.eye(16)
    W3[:] = np.eye(8, 16)
    q = queries([(0, float(u), float(v), float(l)) for u, v, l in
                 zip(*rng.uniform(-2, 2, (2, 200)), rng.uniform(0, 1.5, 200))])
    out, _ = oracle.decode(a, q)
    f = oracle.features(a, q)
    assert np.allclose(out, sigmoid(np.maximum(f[:, :8], 0.0)), atol=1e-15)


@pytest.mark.parametrize("layers,hidden", [(1, 16), (2, 16), (2, 32), (3, 8)])
def test_mlp_equals_dense_torch_evaluation(layers, hidden):
    a, rng = _random_assets(3 + layers, hidden=hidden, out_dim=9, layers=layers)
    q = queries([(0, float(u), float(v), float(l)) for u, v, l in
                 zip(*rng.uniform(-2, 2, (2, 500)), rng.uniform(0, 1.5, 500))])
    out, _ = oracle.decode(a, q)
    x = torch.from_numpy(oracle.features(a, q))
    ps = [torch.from_numpy(p.astype(np.float64)) for p in split_weights(a)]
    h = x
    for l in range(layers):
        h = torch.relu(torch.nn.functional.linear(h, ps[2 * l], ps[2 * l + 1]))
    o = torch.sigmoid(torch.nn.functional.linear(h, ps[-2], ps[-1])).numpy()
    assert np.allclose(out, o, atol=1e-13, rtol=0)


def test_each_query_uses_its_sets_decoder():
    a, rng = _random_assets(11, hidden=16, out_dim=3, num_decoders=3, num_sets=5)
    a.set_to_decoder[:] = [2, 0, 1, 0, 2]
    q = queries([(int(s), float(u), float(v), 0.0) for s, u, v in
                 zip(rng.integers(0, 5, 300), *rng.uniform(-1, 2, (2, 300)))])
    out, _ = oracle.decode(a, q)
    x = torch.from_numpy(oracle.features(a, q))
    for d in range(3):
        ps = [torch.from_numpy(p.astype(np.float64)) for p in split_weights(a, d)]
        h = torch.relu(torch.nn.functional.linear(x, ps[0], ps[1]))
        h = torch.relu(torch.nn.functional.linear(h, ps[2], ps[3]))
        o = torch.sigmoid(torch.nn.functional.linear(h, ps[4], ps[5])).numpy()
        sel = a.set_to_decoder[q["set_id"]] == d
        assert sel.any()
        assert np.allclose(out[sel], o[sel], atol=1e-13)


def test_shared_decoder_equals_one_dense_batch():
    w = W.named("raster-256", "small")
    a = w.assets
    out, _ = oracle.decode(a, w.queries)
    x = torch.from_numpy(oracle.features(a, w.queries))
    ps = [torch.from_numpy(p.astype(np.float64)) for p in split_weights(a, 0)]
    h = torch.relu(torch.nn.functional.linear(x, ps[0], ps[1]))
    h = torch.relu(torch.nn.functional.linear(h, ps[2], ps[3]))
    o = torch.sigmoid(torch.nn.functional.linear(h, ps[4], ps[5])).numpy()
    assert np.allclose(out, o, atol=1e-13)


def test_bad_queries_are_nan_and_counted():
    a, _ = _random_assets(5, num_sets=2, num_decoders=2)
    q = queries([(0, 0.1, 0.2, 0.0), (2, 0.1, 0.2, 0.0), (1, float("nan"), 0.5, 0.0),
                 (1, 0.5, float("inf"), 0.0), (1, 0.5, 0.5, float("nan")), (7, 0.0, 0.0, 0.0)])
    out, bad = oracle.decode(a, q)
    assert bad == 4
    assert np.isfinite(out[0]).all() and np.isfinite(out[4]).all()  # NaN lod counts as 0
    assert np.isnan(out[[1, 2, 3, 5]]).all()


def test_decode_is_invariant_to_query_order():
    w = W.named("gbuffer-1080p", "small")
    out, _ = oracle.decode(w.assets, w.queries)
    p = np.random.default_rng(0).permutation(len(w.queries))
    out2, _ = oracle.decode(w.assets, w.queries[p])
    assert np.array_equal(out2, out[p])


def test_thread_count_does_not_change_results():
    w = W.named("uniform-4m", "small")
    o1, _ = oracle.decode(w.assets, w.queries[:5000], nthreads=1)
    o2, _ = oracle.decode(w.assets, w.queries[:5000], nthreads=7)
    assert np.array_equal(o1, o2)


# -------------------------------------------------------------- bucketing

def _brute_bucket(dec, D, rows=128):
    perm = [i for d in range(D + 1) for i in range(len(dec)) if dec[i] == d]
    counts = [sum(1 for x in dec if x == d) for d in range(D + 1)]
    tiles, pos = [], 0
    for d in range(D + 1):
        for s in range(0, counts[d], rows):
            tiles.append((d, pos + s, min(rows, counts[d] - s)))
        pos += counts[d]
    return perm, counts, tiles


@pytest.mark.parametrize("n,S,D", [(0, 3, 2), (1, 1, 1), (31, 4, 3), (129, 7, 7), (300, 9, 4),
                                   (1000, 40, 5), (257, 3, 3)])
def test_bucketing_matches_brute_force(n, S, D):
    rng = random.Random(n * 31 + S)
    m = [rng.randrange(D) for _ in range(S)]
    sets = [rng.randrange(S + 2) for _ in range(n)]  # some ids out of range
    perm, counts, offsets, tiles = oracle.bucket(np.array(sets, dtype=np.uint32), m, D, tile_rows=16)
    dec = [m[s] if s < S else D for s in sets]
    bp, bc, bt = _brute_bucket(dec, D, rows=16)
    assert perm.tolist() == bp
    assert counts.tolist() == bc
    assert offsets.tolist() == [sum(bc[:d]) for d in range(D + 1)]
    assert [tuple(t) for t in tiles.tolist()] == bt


def test_bucketing_special_cases():
    n = 1000
    same = oracle.bucket(np.zeros(n, np.uint32), [0], 1)[0]
    assert same.tolist() == list(range(n))
    desc = np.arange(n, dtype=np.uint32)[::-1].copy()
    p = oracle.bucket(desc, np.arange(n), n)[0]
    assert p.tolist() == list(range(n))[::-1]
    # empty decoders produce no tiles
    perm, counts, offsets, tiles = oracle.bucket(np.full(10, 2, np.uint32), [0, 1, 2], 3)
    assert counts.tolist() == [0, 0, 10, 0] and tiles.tolist() == [[2, 0, 10]]


# -------------------------------------------------- divergence (Sec. 2, Eq. 1)

def test_divergence_map_and_score():
    assert oracle.divergence_score(np.ones((4, 7))) == 0.0
    X = np.array([[1, 2], [3, 1]])
    assert oracle.divergence_score(X) == pytest.approx((0 + 1 + 2 + 0) / 4)
    ids = [5] * 32 + [1, 2] * 16 + list(range(32)) + [9] * 7
    assert oracle.divergence_map(ids).tolist() == [1, 2, 32, 1]


@pytest.mark.parametrize("d", [1, 2, 5, 10, 32])
def test_controlled_generator_gives_exactly_d_per_warp(d):
    q = W.queries_controlled(99, 64, 32, d)
    D = oracle.divergence_map(q["set_id"])
    assert (D == d).all()
    assert oracle.divergence_score(D) == d - 1


# ---------------------------------------------------- the paper's own numbers

def test_printed_average_speedups_reproduce():
    g = json.load(open(os.path.join(GOLD, "paper_tables.json")))
    for tab in ("table5", "table6"):
        for clk, row in g[tab].items():
            got = [round(oracle.speedup_percent(row[k], row["shared"]), 2) for k in ("wmma", "fma")]
            assert got == row["avg_speedup_percent"], (tab, clk)


def test_table1_category_sizes_sum_to_dataset_size():
    g = json.load(open(os.path.join(GOLD, "paper_tables.json")))
    assert sum(g["table1_category_counts"].values()) == g["table1_total"] == 586


# ------------------------------------------ map sources (Alg. 2 Stage 2, Table 1)

def test_category_and_random_maps_have_table1_group_sizes():
    gold = json.load(open(os.path.join(GOLD, "paper_tables.json")))
    sizes = list(gold["table1_category_counts"].values())
    assert tuple(sizes) == W.CATEGORY_SIZES
    cat = W.map_category()
    assert len(cat) == gold["table1_total"]
    assert np.array_equal(np.bincount(cat), sizes)
    assert (np.diff(cat.astype(np.int64)) >= 0).all()  # contiguous groups in category order
    rnd = W.map_random_sizes(W.BASE_SEED, W.CATEGORY_SIZES)
    assert np.array_equal(np.bincount(rnd, minlength=11), sizes)
    assert not np.array_equal(rnd, cat)


def _blobs(seed, sizes, dim, sep):
    rng = np.random.default_rng(seed)
    centres = rng.standard_normal((len(sizes), dim)) * sep
    lab = np.repeat(np.arange(len(sizes)), sizes)
    return (centres[lab] + rng.standard_normal((len(lab), dim))).astype(np.float32), lab


def test_kmeans_recovers_well_separated_groups():
    F, lab = _blobs(1, [30, 12, 50, 7, 21], 16, sep=40.0)
    init = [0, 30, 42, 92, 99]  # one start row inside each group
    m, mu, it = oracle.kmeans(F, 5, init)
    assert np.array_equal(m, lab)
    assert it == 2  # the second assignment repeats the first
    for g in range(5):
        assert np.allclose(mu[g], F[lab == g].astype(np.float64).mean(0), rtol=0, atol=1e-12)


def test_kmeans_result_is_a_lloyd_fixed_point():
    rng = np.random.default_rng(7)
    F = rng.standard_normal((300, 12)).astype(np.float32)
    m, mu, it = oracle.kmeans(F, 9, rng.permutation(300)[:9], max_iters=500)
    assert it < 500
    X = F.astype(np.float64)
    d = ((X[:, None, :] - mu[None, :, :]) ** 2).sum(-1)  # brute force, every pair
    assert np.array_equal(m, d.argmin(1))
    for g in range(9):
        assert np.allclose(mu[g], X[m == g].mean(0), rtol=0, atol=1e-12)


def test_kmeans_objective_never_increases():
    rng = np.random.default_rng(3)
    F = rng.standard_normal((200, 6)).astype(np.float32)
    init = rng.permutation(200)[:7]
    X = F.astype(np.float64)
    prev = np.inf
    for t in range(1, 12):
        m, mu, _ = oracle.kmeans(F, 7, init, max_iters=t)
        J = ((X - mu[m]) ** 2).sum()
        assert J <= prev * (1 + 1e-12)
        prev = J


def test_kmeans_special_cases():
    rng = np.random.default_rng(5)
    F = rng.standard_normal((40, 5)).astype(np.float32)
    m, mu, _ = oracle.kmeans(F, 1, [17])
    assert (m == 0).all()
    assert np.allclose(mu[0], F.astype(np.float64).mean(0), rtol=0, atol=1e-12)
    m, mu, it = oracle.kmeans(F, 40, np.arange(40))  # every row its own group
    assert np.array_equal(m, np.arange(40)) and it == 2  # the second assignment repeats the first
    assert np.array_equal(mu, F.astype(np.float64))
    # two identical start rows: every distance ties, so the first assignment
    # puts every row in group 0 (ties go to the smaller index), and the empty
    # group 1 keeps its centroid through the update
    G = np.concatenate([F[:10], F[:1]])
    m, mu, it = oracle.kmeans(G, 2, [0, 10], max_iters=1)
    assert (m == 0).all() and it == 1
    assert np.array_equal(mu[1], G[10].astype(np.float64))
    assert np.allclose(mu[0], G.astype(np.float64).mean(0), rtol=0, atol=1e-12)


def test_kmeans_matches_scikit_learn_lloyd():
    sk = pytest.importorskip("sklearn.cluster")
    for seed, (n, dim, m) in enumerate([(500, 8, 6), (586, 32, 11), (120, 3, 4)]):
        F, _ = _blobs(seed, np.full(m, n // m).tolist(), dim, sep=3.0)
        init = np.random.default_rng(seed).permutation(len(F))[:m]
        ours, mu, _ = oracle.kmeans(F, m, init, max_iters=300)
        km = sk.KMeans(n_clusters=m, init=F[init].astype(np.float64), n_init=1, algorithm="lloyd",
                       max_iter=300, tol=0.0).fit(F.astype(np.float64))
        assert np.array_equal(ours, km.labels_)
        assert np.allclose(mu, km.cluster_centers_, rtol=0, atol=1e-9)


# ------------------- paper-faithful decoder: PE, LeakyReLU, 4-channel grid, A x B

def test_positional_encoding_closed_form():
    # dyadic coordinates where sin and cos of 2 pi 2^k u are known exactly
    a = tiny_assets([[(4, 4)]], channels=4, pe_frequencies=3)
    rows = [(0, 0.25, 0.125, 0.0), (0, 1.25, -0.875, 0.0), (0, 0.0, 0.5, 0.0)]
    f = oracle.features(a, queries(rows))[:, 4:].reshape(3, 3, 4)  # [query][k][sin u, cos u, sin v, cos v]
    def expect(u, v):
        return np.array([[np.sin(2 * np.pi * 2 ** k * u), np.cos(2 * np.pi * 2 ** k * u),
                          np.sin(2 * np.pi * 2 ** k * v), np.cos(2 * np.pi * 2 ** k * v)] for k in range(3)])
    # u = 0.25: sin = 1, 0, 0 and cos = 0, -1, 1 for k = 0, 1, 2 (to rounding of pi)
    assert np.allclose(f[0], expect(0.25, 0.125), atol=1e-15)
    assert np.allclose(f[0][:, 0], [1, 0, 0], atol=1e-15) and np.allclose(f[0][:, 1], [0, -1, 1], atol=1e-15)
    # wrap mode encodes the wrapped coordinate: u = 1.25 -> 0.25, v = -0.875 -> 0.125
    assert np.array_equal(f[1], f[0])
    assert np.allclose(f[2], expect(0.0, 0.5), atol=1e-15)
    # clamp mode encodes the coordinate as given
    c = tiny_assets([[(4, 4)]], channels=4, pe_frequencies=3, address_mode=1)
    fc = oracle.features(c, queries([(0, 1.25, -0.875, 0.0)]))[0, 4:].reshape(3, 4)
    assert np.allclose(fc, expect(1.25, -0.875), atol=1e-14)


def test_four_channel_grid_returns_texel_values_at_centres():
    rng = np.random.default_rng(9)
    lat = rng.standard_normal(16 * 16 * 4).astype(np.float32)
    a = tiny_assets([[(16, 16)]], channels=4, latents=lat)
    ij = rng.integers(0, 16, (100, 2))
    q = queries([(0, (i + 0.5) / 16, (j + 0.5) / 16, 0.0) for i, j in ij])
    f = oracle.features(a, q)
    grid = np.float16(lat).astype(np.float64).reshape(16, 16, 4)
    assert np.array_equal(f, grid[ij[:, 1], ij[:, 0]])


@pytest.mark.parametrize("slope", [0.2, 1.25, -0.1])
def test_leaky_relu_identity_weights_closed_form(slope):
    """Identity weights and zero biases reduce the decoder to the activation
    applied once per hidden layer: x -> x for x > 0, slope * x otherwise.  With
    a negative slope the second layer sees a positive value and leaves it."""
    rng = np.random.default_rng(4)
    dims = [[(8, 8), (4, 4)]]
    _, _, total = W.pyramid_layout(1, dims, 1)
    a = tiny_assets(dims, latents=rng.standard_normal(total * 8).astype(np.float32), hidden=16,
                    out_dim=8, activation=1, leaky_slope=slope)
    a.weights[:] = 0
    W1, b1, W2, b2, W3, b3 = split_weights(a)
    W1[:] = np.eye(16)
    W2[:] = np.eye(16)
    W3[:] = np.eye(8, 16)
    q = queries([(0, float(u), float(v), 0.0) for u, v in rng.uniform(-2, 2, (300, 2))])
    out, _ = oracle.decode(a, q)
    f = oracle.features(a, q)[:, :8]
    s = float(np.float32(slope))
    once = np.where(f > 0, f, s * f)
    twice = np.where(once > 0, once, s * once)  # two hidden layers
    assert (f < 0).any()
    expected = np.where(f > 0, f, s * s * f) if s > 0 else np.where(f > 0, f, s * f)
    assert np.allclose(twice, expected, rtol=1e-14, atol=0.0)
    assert np.allclose(out, sigmoid(twice), atol=1e-15)


@pytest.mark.parametrize("hidden,layers", [(16, 1), (32, 2), (64, 2), (64, 3), (128, 4), (32, 4)])
def test_paper_decoder_equals_dense_torch_evaluation(hidden, layers):
    """A x B ablation shapes with the paper's decoder: 4-channel grid, positional
    encoding, LeakyReLU; against torch.nn.functional in fp64."""
    rng = np.random.default_rng(hidden + layers)
    dims = [[(16, 16)]]
    _, _, total = W.pyramid_layout(1, dims, 2)
    a = tiny_assets(dims, num_mips=2, channels=4, latents=rng.standard_normal(total * 4).astype(np.float32),
                    hidden=hidden, out_dim=9, layers=layers, pe_frequencies=4, activation=1, leaky_slope=0.01)
    a.weights[:] = rng.uniform(-0.4, 0.4, a.weights.shape).astype(np.float32)
    q = queries([(0, float(u), float(v), float(l)) for u, v, l in
                 zip(*rng.uniform(-2, 2, (2, 400)), rng.uniform(0, 1.5, 400))])
    out, _ = oracle.decode(a, q)
    x = torch.from_numpy(oracle.features(a, q))
    assert x.shape[1] == 4 + 16
    ps = [torch.from_numpy(p.astype(np.float64)) for p in split_weights(a)]
    h = x
    for l in range(layers):
        h = torch.nn.functional.leaky_relu(torch.nn.functional.linear(h, ps[2 * l], ps[2 * l + 1]),
                                           negative_slope=float(np.float32(0.01)))
    o = torch.sigmoid(torch.nn.functional.linear(h, ps[-2], ps[-1])).numpy()
    assert np.allclose(out, o, atol=1e-13, rtol=0)
