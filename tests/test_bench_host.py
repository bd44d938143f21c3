"""Host-side pieces of bench.py that decide what a measurement reports: the
algorithmic bytes of a scoring call, the clock record taken during the timed
region (a throttled run must show its reasons) and the ncu traffic figure,
which is reported only for the kernel source it was measured on."""
import bench


def test_algorithmic_bytes_of_the_4096_worker_call():
    # state in (3 x int32 a request) + candidates in (3 x 4 B) + flags and
    # margin (5 B a pair) + argbest (4 B a candidate)
    W, B, C = 4096, 128, 32768
    assert bench.algorithmic_bytes(W, B, C) == 6_291_456 + 393_216 + 671_088_640 + 131_072
    assert bench.algorithmic_bytes(W, B, C) == 677_904_384


def test_clock_summary_reads_clocks_and_reasons():
    idle = "0, 2070, 2070, 900.0 W, 0x0, Not Active, Not Active, Not Active, Not Active\n"
    cap = "0, 1980, 2070, 1400.0 W, 0x4, Not Active, Not Active, Not Active, Active\n"
    hot = "0, 1500, 2070, 1400.0 W, 0x8, Active, Not Active, Not Active, Not Active\n"
    s = bench.clock_summary([idle, idle, cap])
    assert s["sm_mhz"] == 2070.0 and s["sm_max_mhz"] == 2070.0 and s["samples"] == 3
    assert s["reasons"] == ["sw_power_cap"]
    s = bench.clock_summary([idle, hot, "garbage line\n", "0, N/A, 2070, 1, 2, 3, 4, 5, 6\n"])
    assert s["samples"] == 2 and s["sm_mhz"] == (2070.0 + 1500.0) / 2
    assert s["reasons"] == ["hw_slowdown"]
    assert bench.clock_summary([]) is None


def test_profiled_traffic_belongs_to_the_current_kernel():
    """The committed ncu traffic is reported only while the scoring kernel's
    source is the one it was captured on; then it must be of the order of the
    algorithmic bytes (no gross re-reads, nothing skipped)."""
    t = bench.profiled_traffic()
    if t is None:
        return  # the kernel changed since the capture: the line reports null
    algo = bench.algorithmic_bytes(4096, 128, 32768)
    assert 0.5 * algo <= t <= 1.5 * algo
