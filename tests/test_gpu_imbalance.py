"""Windowed load imbalance (Section 3.2, Figure 3(c)) on the CUDA path
against the CPU oracle, element by element through the C ABI: every window's
maximum, its instance and the total must be equal."""

import numpy as np
import pytest
import torch

import oracle
import paper_2607_08565_gb300 as pkg
from synth import running_intervals
from gpu_util import T, make_index

pytestmark = pytest.mark.gpu
KEYS = ("max", "argmax", "sum")


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def _gpu(ix, inst, start, end, window, n_windows, **kw):
    out = ix.window_imbalance(T(np.asarray(inst, np.int32)), T(np.asarray(start, np.int64)),
                              T(np.asarray(end, np.int64)), window, n_windows, **kw)
    return {k: v.cpu().numpy() for k, v in out.items()}


def _assert_equal(g, o, ctx):
    for k in KEYS:
        bad = np.nonzero(g[k] != o[k])[0]
        assert len(bad) == 0, f"{ctx} {k}: {len(bad)} mismatches at {bad[:5]}: gpu {g[k][bad[:5]]} oracle {o[k][bad[:5]]}"


@pytest.mark.parametrize("N", [1, 3, 32, 33, 256])
def test_imbalance_matches_oracle_random(N):
    """Short windows and intervals that start and end on window edges, span
    many windows, have zero length or run past the last window; ties between
    instances are common (few distinct lengths)."""
    rng = np.random.default_rng(N)
    ix = make_index(N, 16, 1)
    for trial in range(8):
        n = int(rng.integers(0, 3000)) if trial else 0
        window = int(rng.choice([1, 2, 5, 16, 1000]))
        nw = int(rng.integers(1, 200))
        span = nw * window
        start = rng.integers(0, span + span // 4 + 1, size=n)
        start[::7] = (start[::7] // window) * window  # on an edge
        end = start + rng.choice([0, 1, window, 3 * window, span], size=n)
        inst = rng.integers(0, N, size=n)
        g = _gpu(ix, inst, start, end, window, nw)
        ix.check()
        _assert_equal(g, oracle.window_imbalance(N, window, nw, inst, start, end), f"N={N} trial={trial}")
    ix.close()


def test_imbalance_on_a_serving_trace():
    """32 instances, 30 s windows, 200,000 requests over ~1.6 hours (the
    shape of Figure 3(c)): equal to the oracle, and the imbalance lies
    between 1 and N."""
    N, window = 32, 30_000
    inst, start, end = running_intervals(200_000, N, seed=3)
    nw = int(start[-1] // window) + 1
    ix = make_index(N, 16, 1)
    g = _gpu(ix, inst, start, end, window, nw)
    ix.check()
    ix.close()
    _assert_equal(g, oracle.window_imbalance(N, window, nw, inst, start, end), "trace")
    busy = g["sum"] > 0
    assert busy.all()
    assert (N * g["max"] >= g["sum"]).all() and (g["max"] <= g["sum"]).all()


def test_imbalance_edge_cases():
    N = 4
    ix = make_index(N, 16, 1)
    inst, start, end = [0, 1, 2, 3, 1], [0, 5, 10, 15, 3], [20, 6, 30, 15, 4]
    # no windows: nothing written
    out = ix.window_imbalance(T(np.asarray(inst, np.int32)), T(np.asarray(start, np.int64)),
                              T(np.asarray(end, np.int64)), 10, 0)
    ix.check()
    assert all(v.numel() == 0 for v in out.values())
    # no requests: every window idle
    g = _gpu(ix, np.zeros(0, np.int32), np.zeros(0, np.int64), np.zeros(0, np.int64), 10, 5)
    ix.check()
    assert not any(g[k].any() for k in KEYS)
    # a worked case: windows of 10 ticks
    g = _gpu(ix, inst, start, end, 10, 4)
    ix.check()
    assert g["sum"].tolist() == [10 + 1 + 1, 10 + 10, 10, 0]
    assert g["max"].tolist() == [10, 10, 10, 0]
    assert g["argmax"].tolist() == [0, 0, 2, 0]
    # invalid requests latch INVALID_ARG and are left out; the rest count
    bad_inst, bad_start, bad_end = [0, N, 1, -1, 2, 3], [0, 0, 5, 0, -2, 9], [20, 5, 25, 5, 4, 8]
    g = _gpu(ix, bad_inst, bad_start, bad_end, 10, 3)
    assert ix.status() == pkg.SMETRIC_ERR_INVALID_ARG
    _assert_equal(g, oracle.window_imbalance(N, 10, 3, [0, 1], [0, 5], [20, 25]), "invalid left out")
    # limits refused before any launch
    args = [T(np.asarray(inst, np.int32)), T(np.asarray(start, np.int64)), T(np.asarray(end, np.int64))]
    tiny = torch.empty(1, dtype=torch.int64, device="cuda")
    for window, nw in ((0, 3), (-5, 3), (pkg.SMETRIC_IMBALANCE_MAX_WINDOW + 1, 3), (1 << 36, (1 << 26) + 1)):
        with pytest.raises(pkg.SmetricError) as e:
            ix.window_imbalance(*args, window, nw, workspace=tiny)
        assert e.value.code == pkg.SMETRIC_ERR_INVALID_ARG, (window, nw)
    small = torch.empty(4 * N - 1, dtype=torch.int64, device="cuda")
    with pytest.raises(pkg.SmetricError) as e:
        ix.window_imbalance(*args, 10, 4, workspace=small)
    assert e.value.code == pkg.SMETRIC_ERR_INVALID_ARG
    ix.check()
    ix.close()


def test_imbalance_full_day_properties():
    """A day at 40 requests/s (3.5M requests, 2,880 windows of 30 s): the
    totals add up to the requests' running time inside the day, and sampled
    windows recomputed directly from the intervals are equal."""
    N, window = 32, 30_000
    inst, start, end = running_intervals(3_456_000, N, seed=4)
    nw = 2_880
    ix = make_index(N, 16, 1)
    g = _gpu(ix, inst, start, end, window, nw)
    ix.check()
    ix.close()
    day = nw * window
    assert int(g["sum"].sum()) == int((np.clip(end, 0, day) - np.clip(start, 0, day)).sum())
    rng = np.random.default_rng(0)
    for w in rng.choice(nw, size=24, replace=False):
        lo, hi = w * window, (w + 1) * window
        ov = np.clip(np.minimum(end, hi) - np.maximum(start, lo), 0, None)
        S = np.bincount(inst, weights=ov, minlength=N).astype(np.int64)
        assert g["sum"][w] == S.sum() and g["max"][w] == S.max() and g["argmax"][w] == S.argmax(), w
