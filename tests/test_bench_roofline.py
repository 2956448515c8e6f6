"""bench.py's roofline arithmetic on the CPU: the algorithmic work of a kernel
is per launch (one radix digit pass, one decode step), and the achieved rate is
that work over the average launch time."""
import bench
from paper_2608_21541_gb300 import workloads as W

PEAKS = dict(hbm=6768.8, tensor=1732.7, source="measured")


def test_sort_pass_work_is_per_launch():
    wl = W.WORKLOADS["C3"]
    work = bench.kernel_work(wl, wl.B_live, "sort_scatter")
    # keys and indices read and written once per pass, except the indices of
    # pass 0 (the token indices themselves): 15 B per key per pass on average
    assert work["bytes"] == wl.units * wl.n * 15
    r = bench.roofline_for("sort_scatter", work, 0.25, PEAKS)
    assert r["bound"] == "hbm"
    assert abs(r["achieved"] - work["bytes"] / 0.25e-3 / 1e9) < 0.1


def test_eval_work_leaves_out_the_last_chunk():
    """curve_eval's main launch covers every 128-rank chunk but the last, which
    has its own launch."""
    wl = W.WORKLOADS["C3"]
    work = bench.kernel_work(wl, wl.B_live, "curve_eval")
    assert work["bytes"] == wl.units * (wl.n - 128) * wl.d * 2
    small = W.WORKLOADS["C1"].with_(n=1000)
    assert bench.kernel_work(small, small.B_live, "curve_eval")["bytes"] == \
        small.units * (1000 - 1000 % 128) * small.d * 2


def test_decode_work_is_one_step():
    wl = W.WORKLOADS["C4"]
    work = bench.kernel_work(wl, wl.B_live, "decode_split")
    assert work["bytes"] == wl.B * wl.L * wl.B_live * wl.d * 2 * 2
    r = bench.roofline_for("decode_split", work, 0.6, PEAKS)
    assert abs(r["frac"] - work["bytes"] / 0.6e-3 / 1e9 / PEAKS["hbm"]) < 1e-4


def test_score_passes_are_tensor_bound_at_full_size():
    wl = W.WORKLOADS["C3"]
    work = bench.kernel_work(wl, wl.B_live, "score_pass1")
    assert work["flops"] == 2.0 * wl.G * wl.w * wl.d * wl.n * wl.units
    r = bench.roofline_for("score_pass1", work, 1.8, PEAKS)
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s"


def test_pass_traffic_scales_with_units():
    """The whole-pass DRAM traffic was counted on 16 units (2 layers x 8 KV
    heads) and is reported for a launch of any number of 131072-token units;
    other workloads report none."""
    wl = W.WORKLOADS["C3"]
    full = bench.measured_pass_traffic(wl)
    two = bench.measured_pass_traffic(wl.with_(L=2))
    assert abs(full - 16 * two) <= 16
    assert bench.compress_roofline(wl, wl.B_live, 10.0, PEAKS)["traffic"] == full
    assert bench.measured_pass_traffic(W.WORKLOADS["C1"]) is None
    assert bench.measured_pass_traffic(wl.with_(n=4096)) is None
