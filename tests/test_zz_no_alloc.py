"""The allocation-free bucketing entry point (ntc_bucket_static).

It serves callers that may not allocate device memory when they sort queries
(an engine that owns all GPU memory and forbids cudaMalloc inside its frame
loop).  Its result must equal the oracle's stable sort by decoder bit for bit,
and the context-based bucketing (ntc_debug_bucket) too, on consecutive calls
that share its static scratch.  This file sorts last so a run that stops at the
first failure has run every other test first.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_27888_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _static_bucket(ntc, a, qd):
    n = qd.shape[0]
    perm = torch.full((n,), -1, dtype=torch.int32, device="cuda")
    srt = torch.zeros((n, 4), dtype=torch.int32, device="cuda")
    m = np.ascontiguousarray(a.set_to_decoder, dtype=np.uint32)
    ntc.ntc_bucket_static(m.ctypes.data, a.num_sets, a.num_decoders, qd.data_ptr(), n, perm.data_ptr(),
                          srt.data_ptr(), torch.cuda.current_stream().cuda_stream)
    return perm, srt


def test_static_bucketing_matches_the_oracle_on_consecutive_calls():
    from paper_2608_27888_gb300 import ntc
    cases = [W.named("gbuffer-1080p", "small", "clustered4"), W.named("uniform-4m", "small"),
             W.named("gbuffer-1080p", "small", "clustered4")]
    for w in cases:  # three calls in a row, different sizes and decoder counts
        qd = ntc.queries_to_device(w.queries)
        perm, srt = _static_bucket(ntc, w.assets, qd)
        torch.cuda.synchronize()
        p, _, _, _ = oracle.bucket(w.queries["set_id"], w.assets.set_to_decoder, w.assets.num_decoders)
        assert np.array_equal(perm.cpu().numpy().astype(np.uint32), p)
        assert torch.equal(srt, qd[perm.long()])
        dec = ntc.Decoder(w.assets, "fp16")
        ref_perm, _, _ = dec.bucket(qd)
        dec.close()
        assert torch.equal(perm, ref_perm)


def test_static_bucketing_at_its_largest_size():
    """4,095 decoders and 64 chunks of 2,048 queries: (4095 + 1) x 64 = 262,144
    per-chunk counts, exactly what the static scratch holds (the offsets fill
    the second half of it to its last word).  Out-of-range set ids form the
    extra bucket.  Equal to the oracle bit for bit, twice in a row."""
    from paper_2608_27888_gb300 import ntc
    from tests.util import QD
    D, n = 4095, 64 * 2048
    rng = np.random.default_rng(23)
    q = np.zeros(n, dtype=QD)
    q["set_id"] = rng.integers(0, D + 40, n)  # ~1 % beyond the map
    m = rng.permutation(D).astype(np.uint32)
    qd = ntc.queries_to_device(q)
    p, _, _, _ = oracle.bucket(q["set_id"], m, D)
    for _ in range(2):
        perm = torch.full((n,), -1, dtype=torch.int32, device="cuda")
        srt = torch.zeros((n, 4), dtype=torch.int32, device="cuda")
        ntc.ntc_bucket_static(m.ctypes.data, D, D, qd.data_ptr(), n, perm.data_ptr(), srt.data_ptr(),
                              torch.cuda.current_stream().cuda_stream)
        torch.cuda.synchronize()
        assert np.array_equal(perm.cpu().numpy().astype(np.uint32), p)
        assert torch.equal(srt, qd[perm.long()])


def test_static_bucketing_rejects_sizes_beyond_its_scratch():
    from paper_2608_27888_gb300 import ntc
    w = W.named("raster-256", "small")
    qd = ntc.queries_to_device(w.queries)
    m = np.zeros(1, dtype=np.uint32)
    n_too_many = 262144 // 4096 * 4096 * 2  # (4095 + 1) * ceil(n / 2048) > 262144
    with pytest.raises(ntc.NtcError, match="static scratch"):
        ntc.ntc_bucket_static(m.ctypes.data, 1, 4095, qd.data_ptr(), n_too_many, qd.data_ptr(),
                              qd.data_ptr(), 0)
