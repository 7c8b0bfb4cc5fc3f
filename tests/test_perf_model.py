"""The performance-model calculator (Section 2) against what the paper's
arithmetic and statements fix (CPU only)."""
import json
import math
import os

import pytest

from paper_2504_06419_gb300 import perf_model as pm

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_context.json")


def test_cost_analysis_numbers():
    """Section 5: the saved decoding units for the printed multipliers."""
    g = json.load(open(GOLDEN))["cost_analysis"]
    u = g["decode_budget_units"]
    assert round(pm.decoding_cost_saved(u, g["multiplier_spire_64_512"]), 2) == g["saved_spire_64_512"]
    assert round(pm.decoding_cost_saved(u, g["multiplier_magicdec_64_512"]), 2) == \
        g["saved_magicdec_64_512"]
    assert round(pm.decoding_cost_saved(u, g["multiplier_spire_llama70b_64_65536"]), 2) == \
        g["saved_spire_llama70b"]
    assert round(pm.decoding_cost_saved(u, g["multiplier_magicdec_llama70b_64_65536"]), 2) == \
        g["saved_magicdec_llama70b"]
    assert pm.decoding_cost_saved(u, 1.0) == 0.0


def test_plain_decoding_is_the_unit():
    """k = 0, tau = 1: one target pass per token, multiplier 1, for any costs."""
    for hoi in (10.0, 300.0):
        dt = pm.iteration_time_multiplier(0, 5.0, 7.0, 3.0, 11.0, 13.0, 17.0, hoi)
        assert dt == 1.0 and pm.throughput_multiplier(1.0, dt) == 1.0


def _quarter_draft(batch, ctx, kv_limit=None):
    # target: 8 layers, draft: its last 2 (same widths), so N_t = 4 N_d and, without a
    # sparse cache, KV_t = 4 KV_d (Section 3.2 and Section 4)
    t = pm.transformer_forward_costs(64e6, 8, 512, 512, batch, ctx)
    d = pm.transformer_forward_costs(16e6, 2, 512, 512, batch, ctx, kv_limit=kv_limit)
    return t, d


@pytest.mark.parametrize("ctx", [512, 4096, 65536])
def test_context_cancels_when_memory_bound(ctx):
    """Section 4: with k = 4, N_t = 4 N_d and a full (non-sparse) draft cache,
    L cancels out of delta_t when memory-bound: delta_t = (4 * 1/4 + 1) / 1 = 2."""
    t, d = _quarter_draft(64, ctx)
    hoi = 1e4        # far into the memory-bound regime
    dt = pm.iteration_time_multiplier(4, d.flops, d.weight_bytes, d.kv_bytes,
                                      t.flops, t.weight_bytes, t.kv_bytes, hoi)
    assert math.isclose(dt, 2.0, rel_tol=1e-12)


def test_hoi_cancels_when_both_memory_bound():
    """Section 2 footnote: HOI matters only in the compute-bound corner."""
    t, d = _quarter_draft(64, 8192, kv_limit=65)
    vals = [pm.iteration_time_multiplier(4, d.flops, d.weight_bytes, d.kv_bytes,
                                         t.flops, t.weight_bytes, t.kv_bytes, hoi)
            for hoi in (1e4, 3e4, 1e6)]
    assert max(vals) - min(vals) < 1e-12


def test_compute_bound_corner():
    """With HOI -> 0 every pass is compute-bound and verification costs k+1
    target passes: delta_t = (k C_d + (k+1) C_t) / C_t."""
    dt = pm.iteration_time_multiplier(4, 2.0, 1.0, 1.0, 8.0, 1.0, 1.0, 1e-9)
    assert math.isclose(dt, (4 * 2.0 + 5 * 8.0) / 8.0)


def test_sparse_draft_cache_pays_off_at_long_context():
    """Section 3.1: a sink + window draft cache has constant size, so at long
    L delta_t approaches 1 + k (N_d + KV_d) / (N_t + KV_t) -> 1 while the full
    draft cache stays at 2 (memory-bound, k = 4)."""
    hoi = 1e4
    prev = None
    for ctx in (1024, 8192, 65536, 1 << 20):
        t, d = _quarter_draft(64, ctx, kv_limit=65)   # sink 1 + window 64 (Section 4)
        dt = pm.iteration_time_multiplier(4, d.flops, d.weight_bytes, d.kv_bytes,
                                          t.flops, t.weight_bytes, t.kv_bytes, hoi)
        want = 1.0 + 4 * (d.weight_bytes + d.kv_bytes) / (t.weight_bytes + t.kv_bytes)
        assert math.isclose(dt, want, rel_tol=1e-12)
        assert prev is None or dt < prev
        prev = dt
    assert prev < 1.01


def test_transformer_costs_by_hand():
    c = pm.transformer_forward_costs(100.0, 2, 8, 4, batch=3, ctx=10, tokens=5, kv_limit=6)
    assert c.flops == 2 * 100 * 3 * 5 + 4 * 2 * 8 * 6 * 3 * 5
    assert c.weight_bytes == 200.0
    assert c.kv_bytes == 2 * 2 * 4 * 6 * 3 * 2


def test_measured_delta_t():
    assert pm.measured_delta_t(4, 1.0, 3.0, 2.0) == 3.5
    assert pm.throughput_multiplier(3.401, 3.5) == pytest.approx(0.9717, abs=1e-4)
