"""Host logic of bench.py that its JSON line rests on, without a GPU: the
algorithmic bytes and FLOPs per query behind the roofline, the mean number of
distinct decoders per 32-query warp behind Eq. 1's score, the bounded CPU
sample and its wording.  Each is checked against a closed form or a brute
force written out here, not against bench.py's own formula."""
import numpy as np
import pytest

import bench
from paper_2608_27888_gb300 import workloads as W


@pytest.mark.parametrize("name,variant,bytes_q,flops_q", [
    # 16 B record + 2 levels x 4 taps x 8 fp16 channels + 8 fp32 outputs;
    # 2 x (16*64 + 64*64 + 64*8) MACs
    ("uniform-4m", None, 16 + 2 * 4 * 8 * 2 + 8 * 4, 2 * (16 * 64 + 64 * 64 + 64 * 8)),
    # 9 outputs
    ("gbuffer-2160p", "16", 16 + 2 * 4 * 8 * 2 + 9 * 4, 2 * (16 * 64 + 64 * 64 + 64 * 9)),
    # trilinear: every tap of both mips; H = 128
    ("gbuffer-2160p-x4-trilinear", None, 16 + 2 * 2 * 4 * 8 * 2 + 9 * 4, 2 * (16 * 128 + 128 * 128 + 128 * 9)),
])
def test_algorithmic_bytes_and_flops_per_query(name, variant, bytes_q, flops_q):
    w = W.named(name, "small", variant)
    bpq, flops, w_bytes = bench.shape_costs(w.assets, w.queries)
    assert bpq == bytes_q
    assert flops == flops_q
    a = w.assets
    per_decoder = (a.in_dim * a.hidden + a.hidden * a.hidden + a.hidden * a.out_dim) * 2  # fp16
    assert w_bytes == a.num_decoders * per_decoder


def test_mean_distinct_decoders_per_warp_by_brute_force():
    rng = np.random.default_rng(3)

    class A:
        set_to_decoder = rng.integers(0, 7, 40).astype(np.uint32)

    q = np.zeros(32 * 50 + 13, dtype=W.QUERY_DTYPE)  # a ragged tail is ignored
    q["set_id"] = rng.integers(0, 40, len(q))
    want = np.mean([len({int(A.set_to_decoder[s]) for s in q["set_id"][32 * g:32 * g + 32]}) for g in range(50)])
    assert bench.mean_distinct(q, A) == pytest.approx(want)
    q["set_id"] = 5  # one decoder everywhere: Eq. 1's score 0
    assert bench.mean_distinct(q, A) == 1.0


def test_cpu_sample_of_the_headline_batch():
    q = np.zeros(33_177_600, dtype=np.uint8)
    s, stride = bench.cpu_sample(q)
    assert stride == 33_177_600 // 2 ** 20 == 31
    assert len(s) == -(-33_177_600 // 31)  # every 31st query, from the first
    small = np.zeros(1000, dtype=np.uint8)
    assert bench.cpu_sample(small)[1] == 1


@pytest.mark.parametrize("k,want", [(1, "1st"), (2, "2nd"), (3, "3rd"), (4, "4th"), (11, "11th"), (12, "12th"),
                                    (13, "13th"), (21, "21st"), (22, "22nd"), (31, "31st"), (111, "111th"),
                                    (102, "102nd")])
def test_ordinal(k, want):
    assert bench.ordinal(k) == want
