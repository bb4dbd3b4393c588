"""The paper's two analytical models, fed by counters this library measures.

* Flash lifetime, Eq. (1) (Section 2, "High bandwidth flash"): the writable
  budget of the cold tier is its capacity C times the rated program/erase
  cycles N_PE, and T_life = C * N_PE / (R_W * WAF) is how long that budget
  lasts at the write rate R_W amplified by the write-amplification factor WAF.
* Read power (Section 4, "Methodology"): the sum over memory tiers of each
  tier's read rate times its energy per bit. Serving the hot set from flash
  instead of HBM costs (E_flash - E_HBM) * (hot-set read rate) more.
* Session capacity (Section 4, "Capacity and latency"): the memory left for
  KV (HBM minus the resident weights, plus the cold tier when there is one)
  divided by the mean KV a resident session holds.

The counters come from a trace run: bytes written to the cold tier by pauses
and evictions, bytes decode read from the hot set, and the simulated time the
trace covers (steps x seconds per step).
"""
from __future__ import annotations

SECONDS_PER_YEAR = 365.25 * 24 * 3600
GIB = 1024 ** 3
TIB = 1024 ** 4

# Parameters the paper uses for its modelled HBF tier (Section 4).
HBF_CAPACITY_BYTES = 3 * TIB
HBF_PE_CYCLES = 100_000
HBF_WAF = 1.02
HBM_PJ_PER_BIT = 3.5
WEIGHT_BYTES = 56.8 * GIB          # Qwen3-Coder-30B-A3B bf16 weights, kept in HBM (Section 4)
PAPER_HBM_BYTES = 192 * GIB        # the modelled node's HBM (Section 4)


def lifetime_seconds(write_rate_bytes_per_s: float, capacity_bytes: float = HBF_CAPACITY_BYTES,
                     pe_cycles: float = HBF_PE_CYCLES, waf: float = HBF_WAF) -> float:
    """Eq. (1): T_life = C * N_PE / (R_W * WAF); infinite when nothing is written."""
    if write_rate_bytes_per_s <= 0:
        return float("inf")
    return capacity_bytes * pe_cycles / (write_rate_bytes_per_s * waf)


def lifetime_years(write_rate_bytes_per_s: float, **kw) -> float:
    return lifetime_seconds(write_rate_bytes_per_s, **kw) / SECONDS_PER_YEAR


def read_power_watts(read_rates_bytes_per_s: dict, pj_per_bit: dict) -> float:
    """Sum over tiers of read rate (bytes/s) x 8 bits x energy (pJ/bit)."""
    return sum(rate * 8 * pj_per_bit[tier] * 1e-12 for tier, rate in read_rates_bytes_per_s.items())


def hot_set_power_gap_watts(hot_read_rate_bytes_per_s: float, flash_pj_per_bit: float,
                            hbm_pj_per_bit: float = HBM_PJ_PER_BIT) -> float:
    """Extra read power when the hot set is served from flash instead of HBM."""
    return read_power_watts({"flash": hot_read_rate_bytes_per_s}, {"flash": flash_pj_per_bit}) - \
        read_power_watts({"hbm": hot_read_rate_bytes_per_s}, {"hbm": hbm_pj_per_bit})


def session_capacity(mean_session_bytes: float, hbm_bytes: float,
                     weight_bytes: float = WEIGHT_BYTES, cold_tier_bytes: float = 0.0) -> float:
    """Concurrent sessions whose KV fits in HBM (and the cold tier, if any)
    next to the weights, at a mean resident footprint per session."""
    return (hbm_bytes - weight_bytes + cold_tier_bytes) / mean_session_bytes


def from_trace(cold_write_bytes: float, hot_read_bytes: float, cold_read_bytes: float,
               simulated_seconds: float, flash_pj_per_bit: float = 20.0,
               mean_session_bytes: float | None = None, hbm_bytes: float | None = None) -> dict:
    """Lifetime and read power of one GPU under a measured trace; with the
    trace's mean resident KV per session and the GPU's HBM size, also the
    sessions that fit with HBM alone and with the cold tier added."""
    rw = cold_write_bytes / simulated_seconds
    hot = hot_read_bytes / simulated_seconds
    cold = cold_read_bytes / simulated_seconds
    return {
        "cold_write_rate_gbs": rw / 1e9,
        "hbf_lifetime_years": lifetime_years(rw),
        "hot_read_rate_gbs": hot / 1e9,
        "cold_read_rate_gbs": cold / 1e9,
        "read_power_w_tiered": read_power_watts({"hbm": hot, "flash": cold},
                                                {"hbm": HBM_PJ_PER_BIT, "flash": flash_pj_per_bit}),
        "read_power_w_all_from_flash": read_power_watts({"flash": hot + cold},
                                                        {"flash": flash_pj_per_bit}),
        "flash_pj_per_bit": flash_pj_per_bit,
    } | ({} if mean_session_bytes is None or hbm_bytes is None else {
        "mean_session_gib": mean_session_bytes / GIB,
        "sessions_hbm_only": session_capacity(mean_session_bytes, hbm_bytes),
        "sessions_with_cold_tier": session_capacity(mean_session_bytes, hbm_bytes,
                                                    cold_tier_bytes=HBF_CAPACITY_BYTES),
    })
