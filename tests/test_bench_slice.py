"""The oracle slice that `bench.py` times for its cpu_baseline and its
reference arm (host only, no GPU): the fixed sample (draft step 1 in every
decoder layer, the verify attention of 1 verify layer), the bytes it is
credited with (the same accounting as the GPU arm's draft and verify calls),
and the labelled extrapolation of a round."""

import math

import numpy as np

import bench
from workloads import WORKLOADS, gen


def test_slice_bytes_and_description_workload1():
    wl = WORKLOADS[1]
    sl = bench.OracleSlice(wl)
    lens = gen.ctx_lens(wl)
    k_b = gen.round_plan(wl, 0)[0]
    R = wl.row_bytes
    qo = wl.hq * wl.head_dim * 6 + wl.hq * 4
    assert sl.draft_bytes == len(wl.dec_layers) * sum((int(L) + 1) * R + qo for L in lens)
    assert sl.verify_bytes == sum((int(L) + int(k) + 1) * R + (int(k) + 1) * qo
                                  for L, k in zip(lens, k_b))
    # the GPU arm credits the same bytes to its first draft step and a verify call
    assert sl.draft_bytes == sum(bench.attn_call_bytes(wl, "draft", (1, l), lens, k_b)
                                 for l in wl.dec_layers)
    assert sl.verify_bytes == bench.attn_call_bytes(wl, "verify", wl.dec_layers[0], lens, k_b)
    td, tv = sl.run()
    assert td > 0 and tv > 0
    d = sl.describe(td, tv, 1)
    assert math.isclose(d["value"], sl.bytes / (td + tv) / 1e9)
    assert "1 of 1 verify layers" in d["sample"] and d["kind"] == "oracle"
    assert math.isclose(d["round_us_extrapolated"],
                        round(1e6 * (td * int(k_b.max()) + tv * wl.n_layers), 1), rel_tol=1e-9)
    assert "extrapolated" in d["extrapolation"]
    assert d["cores"] >= 1


def test_slice_sample_names_one_of_28_layers():
    wl = WORKLOADS[2]
    sl = bench.OracleSlice(wl)
    d = sl.describe(1.0, 2.0, 3)
    assert "1 of 28 verify layers" in d["sample"] and "median of 3" in d["sample"]
    assert np.isclose(d["slice_us"], 3e6)
