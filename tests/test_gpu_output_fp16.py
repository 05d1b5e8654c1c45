"""GPU parity of the fp16 output rows (NTC_OUTPUT_FP16; Sec. 4.4's fp16 kernels
write fp16 end to end) through the C ABI.

The rows are the kernel's fp32 sigmoid rounded to nearest even, so they must
equal the fp32-row decode of the same context shape rounded by torch's
round-to-nearest-even bit for bit, on the standard tcgen05 kernel (H = 64 and
128, every small workload, and the full-size headline workload in the
benchmark's launch configuration) and on the general-shape kernel.  Against the
oracle rounded to fp16 they are within the tensor-core tolerance plus one fp16
spacing on [0.5, 1] (2^-11).
"""
import functools

import numpy as np
import pytest
import torch

import oracle
from paper_2608_27888_gb300 import workloads as W

pytestmark = pytest.mark.gpu

TC_MAX, TC_MEAN = 2e-2, 2e-3
HALF_STEP = 2.0 ** -11  # spacing of fp16 on [0.5, 1): the outputs are sigmoids
SMALL = [("raster-256", None), ("uniform-4m", None), ("gbuffer-1080p", "identity"),
         ("gbuffer-1080p", "clustered4"), ("gbuffer-1080p", "shared"), ("gbuffer-2160p", "128"),
         ("gbuffer-2160p", "1"), ("gbuffer-2160p-x4-trilinear", None)]


def ntc():
    from paper_2608_27888_gb300 import ntc as m
    return m


@functools.lru_cache(maxsize=None)
def small(name, variant=None):
    return W.named(name, "small", variant)


def dq(q):
    return ntc().queries_to_device(q)


def rounded_equal(out16, out32):
    """fp16 rows == fp32 rows rounded to nearest even, NaN rows included."""
    assert out16.dtype == torch.float16 and out32.dtype == torch.float32
    a = out16.view(torch.int16).cpu().numpy()
    b = out32.to(torch.float16).view(torch.int16).cpu().numpy()
    return np.array_equal(a, b)


@pytest.mark.parametrize("precision", ["fp16", "bf16"])
@pytest.mark.parametrize("name,variant", SMALL)
def test_fp16_rows_are_the_fp32_rows_rounded(name, variant, precision):
    w = small(name, variant)
    q = dq(w.queries)
    d32 = ntc().Decoder(w.assets, precision)
    d16 = ntc().Decoder(w.assets, precision, output="fp16")
    out32, out16 = d32.decode(q), d16.decode(q)
    assert rounded_equal(out16, out32)
    ref, _ = oracle.decode(w.assets, w.queries)
    ref16 = ref.astype(np.float16).astype(np.float64)
    err = np.abs(out16.cpu().numpy().astype(np.float64) - ref16)
    assert err.max() <= TC_MAX + HALF_STEP, err.max()
    assert err.mean() <= TC_MEAN + HALF_STEP, err.mean()
    d32.close()
    d16.close()


def test_fp16_rows_full_size_headline():
    """The headline workload at full size, as the benchmark launches it."""
    w = W.named("gbuffer-2160p-x4-trilinear", "full")
    q = dq(w.queries)
    d32 = ntc().Decoder(w.assets, "fp16")
    d16 = ntc().Decoder(w.assets, "fp16", output="fp16")
    out32 = d32.decode(q)
    d32.close()
    out16 = d16.decode(q)
    assert rounded_equal(out16, out32)
    # sampled rows against the oracle
    rows = np.random.default_rng(5).choice(len(w.queries), 4096, replace=False)
    ref, _ = oracle.decode(w.assets, w.queries[rows])
    got = out16[torch.from_numpy(rows).to(out16.device)].cpu().numpy().astype(np.float64)
    assert np.abs(got - ref.astype(np.float16).astype(np.float64)).max() <= TC_MAX + HALF_STEP
    # through host buffers: 32 pipelined chunks of ceil(n / 32) queries rounded
    # up to the bucketing chunk, the last one ragged
    hq = torch.from_numpy(np.ascontiguousarray(w.queries).view(np.int32).reshape(-1, 4)).pin_memory()
    host = d16.decode_host(hq)
    assert torch.equal(host.view(torch.int16), out16.cpu().view(torch.int16))
    d16.close()


def test_fp16_rows_of_bad_queries_are_nan_and_counted():
    w = small("uniform-4m")
    q = w.queries[:5000].copy()
    q["set_id"][::97] = 999
    q["u"][5::101] = np.nan
    nbad = len(set(range(0, 5000, 97)) | set(range(5, 5000, 101)))
    dec = ntc().Decoder(w.assets, "fp16", output="fp16")
    got = dec.decode(dq(q))
    bits = got.view(torch.int16).cpu().numpy().astype(np.uint16)
    bad = np.zeros(len(q), dtype=bool)
    bad[::97] = True
    bad[5::101] = True
    assert (bits[bad] == 0x7E00).all()
    assert not np.isnan(got.float().cpu().numpy()[~bad]).any()
    assert dec.error_count() == nbad
    dec.close()


def test_fp16_rows_through_host_buffers():
    w = small("gbuffer-1080p", "identity")
    dec = ntc().Decoder(w.assets, "fp16", output="fp16")
    dev = dec.decode(dq(w.queries))
    hq = torch.from_numpy(np.ascontiguousarray(w.queries).view(np.int32).reshape(-1, 4)).pin_memory()
    host = dec.decode_host(hq)
    assert host.dtype == torch.float16
    assert torch.equal(host.view(torch.int16), dev.cpu().view(torch.int16))
    dec.close()


def test_fp16_rows_of_the_general_shape_kernel():
    w = W.paper_decoder("small")
    q = dq(w.queries)
    d32 = ntc().Decoder(w.assets, "fp16")
    d16 = ntc().Decoder(w.assets, "fp16", output="fp16")
    assert rounded_equal(d16.decode(q), d32.decode(q))
    d32.close()
    d16.close()


def test_fp16_rows_are_bucketed_mode_only():
    w = small("raster-256")
    dec = ntc().Decoder(w.assets, "fp16", output="fp16")
    for mode in ("divergent", "bucketed_mma", "divergent_fma"):
        with pytest.raises(ntc().NtcError) as e:
            dec.decode(dq(w.queries), mode=mode)
        assert e.value.status == 2, mode
    dec.close()
