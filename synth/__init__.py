"""Seeded synthetic agent-serving workloads.

This package is shared by the CUDA path's tests and benchmark and by the CPU
oracle's tests. It produces inputs only: token streams, request offsets,
per-instance loads, index pre-population lists and the replay driver's cache
policy. It contains none of the routing method's arithmetic (no block hashing,
no prefix matching, no cost or argmin).

The production traces the paper studies (Section 3, "Analyzed traces") are
private; the generators here stand in for them with the shapes the paper
reports: >80% KV$ reuse (Finding 1), reuse dominated by follow-up turns of the
same session (Finding 2), a shared system prompt reused by first turns
(Finding 3), and skewed session sizes (Finding 5).
"""

from .traces import (  # noqa: F401
    VOCAB,
    Batch,
    RouteParams,
    AgentTrace,
    BurstTrace,
    agent_trace,
    burst_trace,
    TRACE_CONFIGS,
)
from .replay import ReplayDriver  # noqa: F401
from .intervals import running_intervals  # noqa: F401
