"""The paper's printed context numbers that reports quote are self-consistent
(Section 5 cost analysis) and the bench quotes Table 1's tau unchanged."""
import json
import os

import bench

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_context.json")


def test_cost_analysis_arithmetic():
    g = json.load(open(GOLDEN))["cost_analysis"]
    saved = lambda m: g["decode_budget_units"] * (1 - 1 / m)
    assert round(saved(g["multiplier_spire_64_512"]), 2) == g["saved_spire_64_512"]
    assert round(saved(g["multiplier_magicdec_64_512"]), 2) == g["saved_magicdec_64_512"]
    assert round(g["saved_spire_64_512"] - g["draft_training_cost_units"], 2) == g["net_spire_64_512"]
    assert round(saved(g["multiplier_spire_llama70b_64_65536"]), 2) == g["saved_spire_llama70b"]
    assert round(saved(g["multiplier_magicdec_llama70b_64_65536"]), 2) == g["saved_magicdec_llama70b"]
    assert round(g["saved_spire_llama70b"] - g["draft_training_cost_units"], 2) == g["net_spire_llama70b"]
    # "over 20% more" and "over 16% more" than MagicDec
    assert g["net_spire_64_512"] / g["saved_magicdec_64_512"] > 1.20
    assert g["net_spire_llama70b"] / g["saved_magicdec_llama70b"] > 1.16


def test_bench_quotes_table1_tau():
    g = json.load(open(GOLDEN))["table1_tau_k4"]
    assert bench.SPIRE_TAU_K4_L512 == g["512"]["spire"]
