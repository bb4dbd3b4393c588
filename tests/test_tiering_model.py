"""The paper's lifetime (Eq. 1) and read-power models.

Pinned to figures the paper prints: its 950 W per device at 20 pJ/bit and
its 2.1 / 7.6 / 12.2 kW per 8-GPU node at 8 / 20 / 30 pJ/bit must all follow
from one hot-set read rate under the same power model (Section 4, "Read
energy"); no write means unbounded lifetime (Section 4, "Endurance"); its
165 sessions for HBM alone, 3,900 with a 3 TiB cold tier and the 24x ratio
must follow from its 0.82 GiB mean footprint (Section 4, "Capacity and
latency").
"""
import math

import pytest


@pytest.fixture(scope="module")
def tm():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_25782_gb300 import tiering_model
    return tiering_model


def test_eq1_definition_and_units(tm):
    rw = 0.5e9
    t = tm.lifetime_seconds(rw)
    assert math.isclose(t * rw * tm.HBF_WAF, 3 * 2 ** 40 * 100_000, rel_tol=1e-12)
    assert math.isclose(tm.lifetime_years(rw), t / (365.25 * 86400))
    assert tm.lifetime_years(2 * rw) == pytest.approx(tm.lifetime_years(rw) / 2)
    assert tm.lifetime_years(0.0) == float("inf")


def test_paper_power_figures_share_one_read_rate(tm):
    # one device: 950 W gap at 20 pJ/bit -> the hot-set read rate
    rate = 950.0 / ((20.0 - tm.HBM_PJ_PER_BIT) * 8e-12)
    assert 7.0e12 < rate < 7.4e12          # about HBM speed: the hot set streams every step
    for pj, node_kw in ((8.0, 2.1), (20.0, 7.6), (30.0, 12.2)):
        gap = 8 * tm.hot_set_power_gap_watts(rate, pj) / 1e3
        assert abs(gap - node_kw) < 0.05, (pj, gap)


def test_from_trace(tm):
    r = tm.from_trace(cold_write_bytes=0, hot_read_bytes=1e12, cold_read_bytes=1e10,
                      simulated_seconds=100.0)
    assert r["hbf_lifetime_years"] == float("inf")
    assert r["hot_read_rate_gbs"] == pytest.approx(10.0)
    tiered = 1e10 * 8 * 3.5e-12 + 1e8 * 8 * 20e-12
    assert r["read_power_w_tiered"] == pytest.approx(tiered)
    assert r["read_power_w_all_from_flash"] > r["read_power_w_tiered"]


def test_paper_capacity_figures(tm):
    mean = 0.82 * tm.GIB                       # resident KV per session, steady state
    hbm_only = tm.session_capacity(mean, tm.PAPER_HBM_BYTES)
    tiered = tm.session_capacity(mean, tm.PAPER_HBM_BYTES, cold_tier_bytes=tm.HBF_CAPACITY_BYTES)
    assert abs(hbm_only - 165) < 1.0           # HBM alone: the paper's 165-session limit
    assert abs(tiered / 3900 - 1) < 0.01       # with the flash tier: its 3,900 sessions
    assert round(tiered / hbm_only) == 24      # the ratio the paper reports, 24x
    # the cold tier adds to what HBM holds; without the weights' share both would be off
    assert abs(tm.HBF_CAPACITY_BYTES / mean / 3900 - 1) > 0.03
    assert tm.session_capacity(mean, tm.PAPER_HBM_BYTES, weight_bytes=0) > 230


def test_from_trace_capacity(tm):
    r = tm.from_trace(cold_write_bytes=0, hot_read_bytes=1e12, cold_read_bytes=0,
                      simulated_seconds=1.0, mean_session_bytes=1.0 * tm.GIB,
                      hbm_bytes=tm.PAPER_HBM_BYTES)
    assert r["mean_session_gib"] == pytest.approx(1.0)
    assert r["sessions_hbm_only"] == pytest.approx(192 - 56.8)
    assert r["sessions_with_cold_tier"] == pytest.approx(192 - 56.8 + 3072)
    assert "sessions_hbm_only" not in tm.from_trace(0, 1, 0, 1.0)
