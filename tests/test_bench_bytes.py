"""The roofline arithmetic of bench.py on CPU: algorithmic bytes per call,
written out by hand from their definitions (every visible K/V byte once, the
query in, the fp32 output, the block-table entries and the lengths read), the
per-CTA balance summary and the whole-job value."""
import numpy as np

import bench
import workloads as wl


def test_verify_bytes_uniform8k_by_hand():
    # B=64, L=8192, k=4, 32/8 heads, D=128
    kv = 64 * 8192 * 2 * 8 * 128 * 2          # K and V, bf16
    q_out = 64 * 5 * 32 * 128 * (2 + 4)       # bf16 in, fp32 out
    meta = 64 * (8192 // 64) * 4 + 64 * 4     # block-table entries, ctx_lens
    assert kv == 2_147_483_648
    assert bench.verify_bytes([8192] * 64, 4, 32, 8, 128) == kv + q_out + meta == 2_155_380_992


def test_verify_bytes_ragged_tail_pages():
    # a partial last page still costs one table entry; only visible keys count
    L = [1, 64, 65, 1000]
    pages = 1 + 1 + 2 + 16
    want = sum(L) * 4 * 2 * 64 + 4 * 2 * 8 * 64 * 6 + pages * 4 + 4 * 4
    assert bench.verify_bytes(L, 1, 8, 2, 64) == want


def test_draft_bytes_uniform_step_by_hand():
    # t >> S = 16 + 512: every sequence reads all 528 slots
    t = np.full(64, 8188)
    want = 64 * 528 * 2 * 8 * 128 * 2 + 64 * 32 * 128 * 6 + 64 * 4
    assert bench.draft_bytes(t, 528, 32, 8, 128) == want == 139_985_152
    # short sequences read only their t visible slots
    assert bench.draft_bytes([3, 600], 528, 4, 1, 64) == (3 + 528) * 4 * 64 + 2 * 4 * 64 * 6 + 8


def test_ragged_and_big_workload_bytes():
    L = wl.sample_ctx_lens(wl.CONFIGS["ragged"])
    assert int(L.sum()) == 1_541_606 and L.size == 64
    assert bench.verify_bytes(L, 4, 32, 8, 128) == 6_322_379_224
    L = wl.sample_ctx_lens(wl.CONFIGS["big"])
    assert bench.verify_bytes(L, 8, 64, 8, 128) == 26_154_051_092


def test_cta_balance_summary():
    times = [(1000, 11000), (1500, 9500), (1200, 13200)]   # ns
    b = bench.cta_balance(times)
    assert b["ctas"] == 3
    assert abs(b["busy_us_mean"] - 10.0) < 1e-12
    assert b["busy_us_max"] == 12.0 and b["busy_us_min"] == 8.0
    assert abs(b["max_over_mean"] - 1.2) < 1e-12
    assert b["start_spread_us"] == 0.5 and b["span_us"] == 12.2


def test_job_value_is_weak_scaling():
    # 320 round tokens per rank in 0.44 ms on each of 4 ranks
    assert abs(bench.job_value(320, 4, 0.44) - 4 * 320 / 0.44e-3) < 1e-6
