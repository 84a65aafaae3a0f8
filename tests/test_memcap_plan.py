"""Host arithmetic of the memory-cap batch sweep (Sec. 4, batch scaling under
fixed memory): per-batch cache bytes against the cache sizes the paper prints,
and the largest-batch rule."""

import pytest

import bench
from paper_2605_30351_gb300 import synth

from test_oracle_pins import _golden


def golden():
    return _golden("paper_cache_sizes.txt")


@pytest.fixture(scope="module")
def wan():
    return synth.workload("wan")


def test_dense_cache_per_batch_is_the_papers_six_gb(wan):
    p = bench.memcap_plan(wan, "dense", 180e9)
    g = golden()
    assert p["cache_bytes_per_batch"] == 30 * wan.slots * g["dense_scalars_per_token"] * 2
    assert p["cache_bytes_per_batch"] / 1e9 == pytest.approx(g["dense_cache_gb_bf16"], rel=0.01)


@pytest.mark.parametrize("d_c,key", [(64, "mem_ratio_dc64"), (128, "mem_ratio_dc128"),
                                     (192, "reduction_factor"), (256, "mem_ratio_dc256"),
                                     (512, "mem_ratio_dc512")])
def test_cache_ratio_matches_printed_compression(wan, d_c, key):
    dense = bench.memcap_plan(wan, "dense", 180e9)["cache_bytes_per_batch"]
    mla = bench.memcap_plan(wan.with_(d_c=d_c), "mla", 180e9)["cache_bytes_per_batch"]
    assert dense / mla == pytest.approx(golden()[key], abs=0.006 * golden()[key])


@pytest.mark.parametrize("budget_gb", [40.0, 180.0, 275.0])
def test_max_batch_is_the_largest_that_fits(wan, budget_gb):
    budget = budget_gb * 1e9
    prev = None
    for layout, w in [("dense", wan)] + [("mla", wan.with_(d_c=d)) for d in (64, 128, 192, 256, 512)]:
        p = bench.memcap_plan(w, layout, budget)
        assert p["bytes_at_max_batch"] <= budget < p["bytes_at_max_batch"] + p["per_batch_bytes"]
        if layout == "dense":
            dense_b = p["max_batch"]
        else:
            assert p["max_batch"] > dense_b
            if prev is not None:
                assert p["max_batch"] <= prev          # larger latents, fewer batch elements
            prev = p["max_batch"]


def test_dense_runs_out_where_the_paper_says(wan):
    # the paper's dense MHA leaves the 180 GB budget at B = 28; the plan counts
    # only the attention path, so it may fit one or two more
    assert 28 <= bench.memcap_plan(wan, "dense", 180e9)["max_batch"] <= 30


def test_zero_budget_gives_zero_batch(wan):
    assert bench.memcap_plan(wan, "mla", 0.0)["max_batch"] == 0
