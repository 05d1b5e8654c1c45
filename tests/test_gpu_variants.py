"""GPU parity of the paper-faithful decoder shapes against the CPU oracle.

Sec. 4's decoder: a 4-channel latent grid concatenated with a positional
encoding, LeakyReLU; the MLP ablation varies A neurons x B layers.  These shapes
run the general tcgen05 decode (bucketed, fp16/bf16: max-abs 2e-2, mean-abs
2e-3) and the general per-lane decode (fp32: 1e-5; divergent FMA).  Taps are
bit-exact and features within 1e-5, as for the standard shape.
"""
import functools

import numpy as np
import pytest
import torch

import oracle
from paper_2608_27888_gb300 import workloads as W

pytestmark = pytest.mark.gpu

FP32_TOL = 1e-5
TC_MAX, TC_MEAN = 2e-2, 2e-3

# (name, paper_decoder keyword arguments): Sec. 4's decoder (A64 x B3), the
# ablation's corners, and general shapes of the 2 x 8-channel input
SHAPES = [
    ("paper", dict()),
    ("A16xB3", dict(hidden=16, layers=2)),
    ("A32xB2", dict(hidden=32, layers=1)),
    ("A64xB4", dict(hidden=64, layers=3)),
    ("A128xB5", dict(hidden=128, layers=4)),
    ("A128xB3", dict(hidden=128, layers=2)),
    ("two_levels_pe_relu", dict(levels=2, channels=8, pe=2, activation=0)),
    ("standard_input_leaky", dict(levels=2, channels=8, pe=0, activation=1)),
    ("one_level_8ch_integer_lod", dict(levels=1, channels=8, pe=8, trilinear=False)),
]


def ntc():
    from paper_2608_27888_gb300 import ntc as m
    return m


@functools.lru_cache(maxsize=None)
def work(name):
    return W.paper_decoder("small", **dict(SHAPES)[name])


@functools.lru_cache(maxsize=None)
def ref(name):
    w = work(name)
    return oracle.decode(w.assets, w.queries)


@functools.lru_cache(maxsize=3)
def decoder(name, precision):
    return ntc().Decoder(work(name).assets, precision)


def dq(q):
    return ntc().queries_to_device(q)


def check_tc(got, ref, what):
    err = np.abs(got.astype(np.float64) - ref)
    assert np.isfinite(got).all(), what
    assert err.max() <= TC_MAX, f"{what}: max abs {err.max():.3e}"
    assert err.mean() <= TC_MEAN, f"{what}: mean abs {err.mean():.3e}"


@pytest.mark.parametrize("name", [s for s, _ in SHAPES])
def test_taps_and_features(name):
    w = work(name)
    dec = decoder(name, "fp16")
    idx, wt, tt = dec.taps(dq(w.queries))
    ri, rw, rt = oracle.taps(w.assets, w.queries)
    assert np.array_equal(idx.cpu().numpy().view(np.uint64), ri)
    assert np.array_equal(wt.cpu().numpy().view(np.uint32), rw.view(np.uint32))
    assert np.array_equal(tt.cpu().numpy().view(np.uint32), rt.view(np.uint32))
    f = dec.features(dq(w.queries)).cpu().numpy()
    rf = oracle.features(w.assets, w.queries)
    assert f.shape == rf.shape == (len(w.queries), w.assets.in_dim)
    assert np.abs(f - rf).max() <= 1e-5 * max(1.0, np.abs(rf).max())


@pytest.mark.parametrize("precision", ["fp16", "bf16"])
@pytest.mark.parametrize("mode", ["bucketed", "divergent_fma"])
@pytest.mark.parametrize("name", [s for s, _ in SHAPES])
def test_tensor_core_precisions(name, mode, precision):
    w = work(name)
    r, _ = ref(name)
    got = decoder(name, precision).decode(dq(w.queries), mode=mode).cpu().numpy()
    check_tc(got, r, f"{name} {mode} {precision}")


@pytest.mark.parametrize("mode", ["bucketed", "divergent_fma"])
@pytest.mark.parametrize("name", [s for s, _ in SHAPES])
def test_fp32_precision(name, mode):
    w = work(name)
    r, _ = ref(name)
    got = decoder(name, "fp32").decode(dq(w.queries), mode=mode).cpu().numpy()
    assert np.abs(got - r).max() <= FP32_TOL


def test_order_invariance_is_bitwise():
    w = work("paper")
    dec = decoder("paper", "fp16")
    out = dec.decode(dq(w.queries)).cpu().numpy()
    p = np.random.default_rng(2).permutation(len(w.queries))
    assert np.array_equal(dec.decode(dq(w.queries[p])).cpu().numpy(), out[p])


@pytest.mark.parametrize("n", [1, 127, 128, 129, 5001])
def test_bad_queries_and_ragged_sizes(n):
    w = work("paper")
    q = np.resize(w.queries, n).copy()
    q["set_id"][::7] = 1000
    q["u"][3::11] = np.inf
    r, nbad = oracle.decode(w.assets, q)
    for prec, mode in (("fp16", "bucketed"), ("fp32", "bucketed"), ("bf16", "divergent_fma")):
        dec = decoder("paper", prec)
        dec.reset_error_count()
        got = dec.decode(dq(q), mode=mode).cpu().numpy()
        assert np.array_equal(np.isnan(got), np.isnan(r)), (prec, mode)
        ok = ~np.isnan(r).any(1)
        tol = FP32_TOL if prec == "fp32" else TC_MAX
        assert np.abs(got[ok] - r[ok]).max(initial=0.0) <= tol, (prec, mode)
        assert dec.error_count() == nbad
        dec.reset_error_count()


def test_modes_without_a_general_kernel_are_refused():
    m = ntc()
    w = work("paper")
    dec = decoder("paper", "fp16")
    for mode in ("divergent", "bucketed_mma"):
        with pytest.raises(m.NtcError, match="decoder shape"):
            dec.decode(dq(w.queries[:64]), mode=mode)
    torch.cuda.synchronize()


@pytest.mark.parametrize("slope", [1.25, -0.1])
def test_leaky_slopes_outside_the_unit_interval(slope):
    """A LeakyReLU slope outside [0, 1] takes the kernels' general activation
    (a select, not max(x, slope * x)); every precision and mode agrees with the
    oracle."""
    w = W.paper_decoder("small", leaky_slope=slope)
    r, _ = oracle.decode(w.assets, w.queries)
    for precision in ("fp16", "bf16", "fp32"):
        dec = ntc().Decoder(w.assets, precision)
        for mode in ("bucketed", "divergent_fma"):
            got = dec.decode(dq(w.queries), mode=mode).cpu().numpy()
            if precision == "fp32":
                assert np.abs(got - r).max() <= FP32_TOL, (precision, mode)
            else:
                check_tc(got, r, f"slope {slope} {mode} {precision}")
        dec.close()
