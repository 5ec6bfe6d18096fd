"""Host logic of bench.py's router-vs-exact saliency report (CPU): the rank correlation
against scipy's Spearman, the routing of a saliency against the oracle's §4.2 rule, and the
route table's bookkeeping, and the roofline's fraction of the burst peak."""
import numpy as np
import pytest
from scipy.stats import spearmanr

import bench
import oracle


@pytest.mark.parametrize("seed", range(5))
def test_rank_correlation_is_spearman(seed):
    g = np.random.default_rng(seed)
    a = g.standard_normal(16)
    b = a + g.standard_normal(16) * (0.2 * seed)
    b[3] = b[7]  # a tie
    assert np.isclose(bench.rank_correlation(a, b), spearmanr(a, b).statistic, atol=1e-12)
    assert np.isclose(bench.rank_correlation(a, a), 1.0)
    assert np.isclose(bench.rank_correlation(a, -a), -1.0)


def test_route_of_follows_the_routing_equation():
    for s in [0.0, 0.005, 0.01, np.nextafter(np.float32(0.01), np.float32(1)), 0.05, 0.2,
              np.nextafter(np.float32(0.2), np.float32(0)), 0.7, 1.0, float("nan")]:
        assert bench.route_of(s) == oracle.select_mode(s), s


def test_saliency_agreement_table():
    s_router = [0.001, 0.05, 0.5, 0.3, 0.002]
    s_exact = [0.002, 0.005, 0.9, 0.1, 0.003]
    rep = bench.saliency_agreement(s_router, s_exact)
    assert rep["routes_router"] == [0, 1, 2, 2, 0]
    assert rep["routes_exact"] == [0, 0, 2, 1, 0]
    assert rep["route_table"] == [[2, 0, 0], [1, 0, 0], [0, 1, 1]]
    assert rep["routes_agree"] == 3
    assert np.isclose(rep["spearman"], spearmanr(s_router, s_exact).statistic)


def test_burst_fraction_of_the_roofline():
    pk = {"bf16_tflops": 2000.0, "bf16_tflops_sustained": 1600.0,
          "clocks_under_load": {"sm_mhz_median": 1500.0}}
    out = bench.burst_fraction(pk, 1200.0)
    assert out == {"peak_burst": 2000.0, "frac_of_burst": 0.6, "peak_sustained_sm_mhz": 1500.0}
    assert bench.burst_fraction({}, 1200.0) == {}
    assert bench.burst_fraction({"bf16_tflops": 1000.0}, 500.0) == {"peak_burst": 1000.0,
                                                                      "frac_of_burst": 0.5}
