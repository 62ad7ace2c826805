import os
"""Host-side helpers of bench.py (no GPU): the mean accepted tokens reported from an
acceptance histogram, the clock-sample summary that decides whether a run is kept, and the
digest that ties the committed DRAM-traffic record to the kernel code."""

import numpy as np

import bench
from oracle import alr_oracle as orc


def test_mat_from_histogram_matches_per_anchor_mean():
    """MAT (Sec. 4) is the mean over anchors of accepted slots + 1; from the histogram of the
    oracle's accepted lengths it must equal the direct per-anchor mean."""
    rng = np.random.default_rng(4)
    A, B = 300, 16
    am_t = rng.integers(0, 3, A * B)
    am_d = np.where(rng.random(A * B) < 0.8, am_t, rng.integers(0, 3, A * B))
    acc, hist = orc.accept_len(am_d, am_t, B)
    assert abs(bench.mean_accepted_tokens(hist.tolist()) - (acc.mean() + 1.0)) < 1e-12
    assert bench.mean_accepted_tokens([0] * (B + 1)) is None
    assert bench.mean_accepted_tokens([5, 0, 0]) == 1.0


def test_clock_samples_summary_and_throttle_reasons():
    """nvidia-smi lines in the sampler's column order: idle edge samples do not count toward
    the median, every reason seen active is reported, malformed lines are skipped."""
    row = "0, {sm}, 2070, 1370.5, 0x{act}, {hw}, {hwt}, {swt}, {cap}\n"
    lines = [row.format(sm=345, act="0", hw="Not Active", hwt="Not Active", swt="Not Active",
                        cap="Not Active"),
             row.format(sm=1600, act="4", hw="Not Active", hwt="Not Active", swt="Not Active",
                        cap="Active"),
             row.format(sm=1650, act="4", hw="Not Active", hwt="Not Active", swt="Not Active",
                        cap="Active"),
             row.format(sm=1620, act="8", hw="Active", hwt="Not Active", swt="Not Active",
                        cap="Not Active"),
             "garbage line\n", "0, [N/A], 2070, 0, 0x0, a, b, c, d\n"]
    c = bench.parse_clocks(lines)
    assert c["sm_mhz"] == 1620.0 and c["sm_max_mhz"] == 2070.0
    assert c["reasons"] == ["hw_slowdown", "sw_power_cap"]
    assert c["samples"] == 4
    assert bench.parse_clocks(["garbage\n"]) is None


def test_traffic_record_follows_kernel_code_not_comments():
    """The DRAM-traffic record of a kernel is tied to a digest of its sources' code: a comment
    or a blank line leaves it valid, a changed token invalidates it."""
    src = {"a.cu": "int f(int x) {\n  return x + 1;  // add one\n}\n", "b.h": "/* doc */ int g;"}
    names = list(src)
    h0 = bench.kernel_sources_sha256(names, read=lambda rel: src[rel])
    commented = dict(src, **{"a.cu": "// header\nint f(int x) {\n\n"
                                      "  return x + 1; /* one */\n}\n"})
    assert bench.kernel_sources_sha256(names, read=lambda rel: commented[rel]) == h0
    changed = dict(src, **{"a.cu": "int f(int x) {\n  return x + 2;\n}\n"})
    assert bench.kernel_sources_sha256(names, read=lambda rel: changed[rel]) != h0


def test_every_recorded_kernel_names_existing_sources():
    for phase, files in bench.KERNEL_SOURCES.items():
        for rel in files:
            assert os.path.exists(os.path.join(bench.ROOT, rel)), (phase, rel)
