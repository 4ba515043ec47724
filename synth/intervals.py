"""Seeded running intervals of routed requests, for the windowed load
imbalance (Section 3.2, Figure 3(c): load = average running requests per
instance in 30 s windows, 32 instances).

Inputs only: each request's instance and its [start, end) in integer
milliseconds. Arrivals are a Poisson process whose rate follows a slow
diurnal-style swing; a request runs for a log-normal time (prefill plus
decode of an agent turn, median ~8 s, a heavy tail to minutes); instances
are drawn from a skewed distribution that drifts over the trace, so some
windows are balanced and others are not.
"""

from __future__ import annotations

import numpy as np


def running_intervals(n_requests: int, num_instances: int = 32, seed: int = 0, rate_per_s: float = 40.0,
                      median_ms: float = 8000.0, sigma: float = 1.0, skew: float = 0.3):
    """Returns (instance int32, start int64 ms, end int64 ms), in arrival order."""
    rng = np.random.default_rng([0x1B, seed])
    gaps = rng.exponential(1000.0 / rate_per_s, size=n_requests)
    t = np.cumsum(gaps)
    # the arrival rate swings by about +-25 % over a period of ~6.3 hours
    t = t + 0.25 * 3.6e6 * np.sin(t / 3.6e6)
    start = np.maximum(np.floor(t), 0).astype(np.int64)
    start.sort()
    dur = np.floor(rng.lognormal(np.log(median_ms), sigma, size=n_requests)).astype(np.int64)
    end = start + dur
    # instance weights: a power law whose ranking rotates every ~10 minutes
    ranks = np.arange(1, num_instances + 1, dtype=np.float64) ** -skew
    epoch = start // 600_000
    shift = (epoch * 7) % num_instances
    pick = rng.choice(num_instances, size=n_requests, p=ranks / ranks.sum())
    inst = ((pick + shift) % num_instances).astype(np.int32)
    return inst, start, end
