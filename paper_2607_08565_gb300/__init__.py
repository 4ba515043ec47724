"""Python binding of libsmetric.so, the GB300 batched routing path of
balanced session-centric scheduling (SMetric, arXiv 2607.08565).

Functions carry the C ABI's names and only marshal arguments: device arrays
may be passed as torch tensors or raw device pointers (ints); streams as a
torch.cuda.Stream, a raw cudaStream_t (int) or None for torch's current
stream. Every computation runs in the library's CUDA kernels; there is no
CPU fallback, and using the binding without the built library raises.

SMetricIndex wraps one index and allocates output tensors for convenience.
"""

from __future__ import annotations

import ctypes as C
import os
from typing import Optional

from .build_lib import LIB as _LIB_PATH

SMETRIC_OK = 0
SMETRIC_ERR_INVALID_ARG = -1
SMETRIC_ERR_OOM = -2
SMETRIC_ERR_TABLE_FULL = -3
SMETRIC_ERR_CUDA = -4
SMETRIC_ERR_OVERFLOW = -5
SMETRIC_ERR_TOO_LARGE = -6
SMETRIC_NOALLOC_MAX_REQUESTS = 4096
SMETRIC_NOALLOC_MAX_BLOCKS = 32768
SMETRIC_MAX_INSTANCES = 256
SMETRIC_MAX_WEIGHT = 1 << 20
SMETRIC_MAX_LOAD = 1 << 40
SMETRIC_MAX_PROBE = 65536
SMETRIC_FLAG_HOST_STAGING = 1
SMETRIC_FLAG_PIPELINE = 2
SMETRIC_POLICY_MAX_LEN = 1 << 24
SMETRIC_POLICY_MAX_QUEUED = 1 << 59
SMETRIC_COMMIT_GLOBAL = 1
SMETRIC_POLICY_MAX_TPOT = 1 << 60
SMETRIC_POLICY_MAX_REQUESTS = 1 << 20
SMETRIC_IMBALANCE_MAX_WINDOW = 1 << 36
SMETRIC_IMBALANCE_MAX_REQUESTS = 1 << 26
SMETRIC_IMBALANCE_MAX_CELLS = 1 << 31
SMETRIC_SCORER_BAILIAN = 1
SMETRIC_SCORER_LMETRIC = 2

EXPORTED = (
    "smetric_index_create", "smetric_index_destroy", "smetric_index_clear",
    "smetric_index_insert", "smetric_index_evict", "smetric_index_lookup",
    "smetric_index_mask_words", "smetric_route_batch", "smetric_block_hashes",
    "smetric_route_batch_host", "smetric_status", "smetric_strerror",
    "smetric_profile_enable", "smetric_profile_read", "smetric_profile_kernel_name",
    "smetric_launch_count", "smetric_block_hashes_noalloc", "smetric_route_batch_policy",
    "smetric_index_commit_batch", "smetric_route_batch_policy_coloc", "smetric_link_sessions",
    "smetric_route_batch_baseline", "smetric_route_batch_sequential", "smetric_reuse_workspace_bytes",
    "smetric_reuse_breakdown", "smetric_imbalance_workspace_bytes", "smetric_window_imbalance",
    "smetric_route_batches", "smetric_index_set_lru", "smetric_index_lru_sizes", "smetric_route_commit_batch",
)


class SmetricError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        super().__init__(f"{where}: {smetric_strerror(code)} ({code})")


class smetric_index_config(C.Structure):
    _fields_ = [
        ("num_instances", C.c_int32),
        ("block_size", C.c_int32),
        ("session_blocks", C.c_int32),
        ("flags", C.c_int32),
        ("capacity_slots", C.c_uint64),
        ("hash_seed", C.c_uint64),
        ("max_batch_requests", C.c_int64),
        ("max_batch_tokens", C.c_int64),
    ]


class smetric_weights(C.Structure):
    _fields_ = [("w_load", C.c_int64), ("w_miss", C.c_int64), ("w_glob", C.c_int64)]


class smetric_policy(C.Structure):
    _fields_ = [("c_lin", C.c_int64), ("c_att", C.c_int64), ("ttft_d0", C.c_int64),
                ("ttft_d1", C.c_int64), ("hit_num", C.c_int64), ("hit_den", C.c_int64),
                ("rr_base", C.c_int32), ("reserved", C.c_int32)]


_lib = None


def library_path() -> str:
    return _LIB_PATH


def lib():
    """The loaded libsmetric.so. Raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError(
                f"libsmetric.so is not built ({_LIB_PATH}); run __graft_entry__.build() "
                "or python -m paper_2607_08565_gb300.build_lib")
        L = C.CDLL(_LIB_PATH)
        P, I32, I64, U64 = C.c_void_p, C.c_int32, C.c_int64, C.c_uint64
        sig = {
            "smetric_index_create": (C.c_int, [C.POINTER(smetric_index_config), C.POINTER(P)]),
            "smetric_index_destroy": (C.c_int, [P]),
            "smetric_index_clear": (C.c_int, [P, P]),
            "smetric_index_insert": (C.c_int, [P, P, P, I64, P]),
            "smetric_index_evict": (C.c_int, [P, P, P, I64, P]),
            "smetric_index_lookup": (C.c_int, [P, P, I64, P, P]),
            "smetric_index_mask_words": (I32, [P]),
            "smetric_route_batch": (C.c_int, [P, P, I64, P, I32, P, smetric_weights, P, P, P, P, P,
                                              I64, P]),
            "smetric_route_batches": (C.c_int, [P, I32, P, P, P, P, P, smetric_weights, P, P, P, P, P]),
            "smetric_route_batch_policy": (C.c_int, [P, P, I64, P, I32, P, P, P, smetric_policy, P, P,
                                                     P, P, P, P, I64, P]),
            "smetric_index_commit_batch": (C.c_int, [P, P, I32, P, P, P, I32, P, P]),
            "smetric_index_set_lru": (C.c_int, [P, I64, I64]),
            "smetric_route_commit_batch": (C.c_int, [P, P, I64, P, I32, P, smetric_weights, P, P, P, P, P, I64,
                                                     I32, P]),
            "smetric_index_lru_sizes": (C.c_int, [P, P, P]),
            "smetric_link_sessions": (C.c_int, [P, P, I64, P, I32, P, P, P, P, P]),
            "smetric_reuse_workspace_bytes": (I64, [I64]),
            "smetric_imbalance_workspace_bytes": (I64, [I32, I32]),
            "smetric_window_imbalance": (C.c_int, [P, P, P, P, I32, I64, I32, P, I64, P, P, P, P]),
            "smetric_reuse_breakdown": (C.c_int, [P, P, I64, P, I32, P, P, P, I64, P, P, P, P, P]),
            "smetric_route_batch_sequential": (C.c_int, [P, P, I64, P, I32, P, smetric_weights, P, P, P, P, P,
                                                         I64, P, P]),
            "smetric_route_batch_baseline": (C.c_int, [P, P, I64, P, I32, I32, P, P, I64, I64, P, P, P, P, P,
                                                       I64, P]),
            "smetric_route_batch_policy_coloc": (C.c_int, [P, P, I64, P, I32, P, P, P, P, P, smetric_policy,
                                                           P, P, P, P, P, P, I64, P]),
            "smetric_block_hashes": (C.c_int, [P, P, I64, P, I32, P, P, I64, P]),
            "smetric_block_hashes_noalloc": (C.c_int, [P, I64, P, I32, I32, I32, C.c_uint64, P, P, I64,
                                                      P, P]),
            "smetric_route_batch_host": (C.c_int, [P, P, I64, P, I32, P, smetric_weights, P, P, P,
                                                   P, P]),
            "smetric_status": (C.c_int, [P, P]),
            "smetric_strerror": (C.c_char_p, [C.c_int]),
            "smetric_profile_enable": (C.c_int, [P, I32]),
            "smetric_profile_read": (C.c_int, [P, I32, P, P]),
            "smetric_profile_kernel_name": (C.c_char_p, [I32]),
            "smetric_launch_count": (I64, [P]),
        }
        for name, (res, args) in sig.items():
            f = getattr(L, name)
            f.restype, f.argtypes = res, args
        _lib = L
    return _lib


# ---------------------------------------------------------------------------
# marshalling helpers
# ---------------------------------------------------------------------------

def _ptr(x) -> Optional[int]:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        if not x.is_contiguous():
            raise ValueError("arrays must be contiguous")
        return x.data_ptr() if x.numel() > 0 else None
    if hasattr(x, "ctypes"):  # numpy array (host memory)
        return x.ctypes.data if x.size > 0 else None
    raise TypeError(f"cannot pass {type(x)} as a pointer")


def _stream(s) -> Optional[int]:
    if s is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(s, int):
        return s
    return s.cuda_stream


def _check(rc: int, where: str):
    if rc != SMETRIC_OK:
        raise SmetricError(rc, where)


def _weights(w) -> smetric_weights:
    if isinstance(w, smetric_weights):
        return w
    a, b, c = w
    return smetric_weights(int(a), int(b), int(c))


# ---------------------------------------------------------------------------
# C ABI, one function per entry point
# ---------------------------------------------------------------------------

def smetric_index_create(cfg: smetric_index_config) -> int:
    h = C.c_void_p()
    _check(lib().smetric_index_create(C.byref(cfg), C.byref(h)), "smetric_index_create")
    return h.value


def smetric_index_destroy(idx: int) -> None:
    _check(lib().smetric_index_destroy(idx), "smetric_index_destroy")


def smetric_index_clear(idx: int, stream=None) -> None:
    _check(lib().smetric_index_clear(idx, _stream(stream)), "smetric_index_clear")


def smetric_index_insert(idx: int, d_keys, d_tiers, n: int, stream=None) -> None:
    _check(lib().smetric_index_insert(idx, _ptr(d_keys), _ptr(d_tiers), n, _stream(stream)),
           "smetric_index_insert")


def smetric_index_evict(idx: int, d_keys, d_tiers, n: int, stream=None) -> None:
    _check(lib().smetric_index_evict(idx, _ptr(d_keys), _ptr(d_tiers), n, _stream(stream)),
           "smetric_index_evict")


def smetric_index_lookup(idx: int, d_keys, n: int, d_masks, stream=None) -> None:
    _check(lib().smetric_index_lookup(idx, _ptr(d_keys), n, _ptr(d_masks), _stream(stream)),
           "smetric_index_lookup")


def smetric_index_mask_words(idx: int) -> int:
    return int(lib().smetric_index_mask_words(idx))


def smetric_route_batch(idx: int, d_tokens, n_tokens: int, d_offsets, n_requests: int, d_load,
                        w, d_instance, d_local_hit, d_global_hit, d_session_key,
                        d_block_hashes=None, hashes_cap: int = 0, stream=None) -> None:
    _check(lib().smetric_route_batch(idx, _ptr(d_tokens), n_tokens, _ptr(d_offsets), n_requests,
                                     _ptr(d_load), _weights(w), _ptr(d_instance), _ptr(d_local_hit),
                                     _ptr(d_global_hit), _ptr(d_session_key), _ptr(d_block_hashes),
                                     hashes_cap, _stream(stream)), "smetric_route_batch")


def smetric_route_commit_batch(idx: int, d_tokens, n_tokens: int, d_offsets, n_requests: int, d_load, w,
                               d_instance, d_local_hit, d_global_hit, d_session_key, d_block_hashes,
                               hashes_cap: int, flags: int = 0, stream=None) -> None:
    _check(lib().smetric_route_commit_batch(idx, _ptr(d_tokens), n_tokens, _ptr(d_offsets), n_requests,
                                            _ptr(d_load), _weights(w), _ptr(d_instance), _ptr(d_local_hit),
                                            _ptr(d_global_hit), _ptr(d_session_key), _ptr(d_block_hashes),
                                            hashes_cap, flags, _stream(stream)), "smetric_route_commit_batch")


def smetric_route_batches(idx: int, d_tokens, n_tokens, d_offsets, n_requests, d_load, w, d_instance,
                          d_local_hit, d_global_hit, d_session_key, stream=None) -> None:
    """Several batches in one call; every argument but idx, w and stream is a
    sequence with one entry per batch (device arrays, or counts)."""
    nb = len(n_requests)
    if not all(len(x) == nb for x in (d_tokens, n_tokens, d_offsets, d_load, d_instance, d_local_hit,
                                      d_global_hit, d_session_key)):
        raise ValueError("every per-batch sequence needs one entry per batch")
    ptrs = lambda xs: (C.c_void_p * max(nb, 1))(*[_ptr(x) for x in xs])
    _check(lib().smetric_route_batches(idx, nb, ptrs(d_tokens), (C.c_int64 * max(nb, 1))(*n_tokens),
                                       ptrs(d_offsets), (C.c_int32 * max(nb, 1))(*n_requests), ptrs(d_load),
                                       _weights(w), ptrs(d_instance), ptrs(d_local_hit), ptrs(d_global_hit),
                                       ptrs(d_session_key), _stream(stream)), "smetric_route_batches")


def _policy(p) -> smetric_policy:
    if isinstance(p, smetric_policy):
        return p
    d = dict(p)
    return smetric_policy(int(d["c_lin"]), int(d["c_att"]), int(d["ttft_d0"]), int(d["ttft_d1"]),
                          int(d["hit_num"]), int(d["hit_den"]), int(d.get("rr_base", 0)), 0)


def smetric_route_batch_policy(idx: int, d_tokens, n_tokens: int, d_offsets, n_requests: int,
                               d_queued, d_turn, d_est_hit, policy, d_instance, d_local_hit,
                               d_global_hit, d_stick, d_session_key, d_block_hashes=None,
                               hashes_cap: int = 0, stream=None) -> None:
    _check(lib().smetric_route_batch_policy(
        idx, _ptr(d_tokens), n_tokens, _ptr(d_offsets), n_requests, _ptr(d_queued), _ptr(d_turn),
        _ptr(d_est_hit), _policy(policy), _ptr(d_instance), _ptr(d_local_hit), _ptr(d_global_hit),
        _ptr(d_stick), _ptr(d_session_key), _ptr(d_block_hashes), hashes_cap, _stream(stream)),
        "smetric_route_batch_policy")


def smetric_route_batch_policy_coloc(idx: int, d_tokens, n_tokens: int, d_offsets, n_requests: int,
                                     d_queued, d_tpot_budget, d_num_requests, d_turn, d_est_hit, policy,
                                     d_instance, d_local_hit, d_global_hit, d_stick, d_session_key,
                                     d_block_hashes=None, hashes_cap: int = 0, stream=None) -> None:
    _check(lib().smetric_route_batch_policy_coloc(
        idx, _ptr(d_tokens), n_tokens, _ptr(d_offsets), n_requests, _ptr(d_queued), _ptr(d_tpot_budget),
        _ptr(d_num_requests), _ptr(d_turn), _ptr(d_est_hit), _policy(policy), _ptr(d_instance),
        _ptr(d_local_hit), _ptr(d_global_hit), _ptr(d_stick), _ptr(d_session_key), _ptr(d_block_hashes),
        hashes_cap, _stream(stream)), "smetric_route_batch_policy_coloc")


def smetric_route_batch_baseline(idx: int, d_tokens, n_tokens: int, d_offsets, n_requests: int, scorer: int,
                                 d_queued, d_batch, lam_num: int, lam_den: int, d_instance, d_local_hit,
                                 d_global_hit, d_session_key, d_block_hashes=None, hashes_cap: int = 0,
                                 stream=None) -> None:
    _check(lib().smetric_route_batch_baseline(
        idx, _ptr(d_tokens), n_tokens, _ptr(d_offsets), n_requests, scorer, _ptr(d_queued), _ptr(d_batch),
        lam_num, lam_den, _ptr(d_instance), _ptr(d_local_hit), _ptr(d_global_hit), _ptr(d_session_key),
        _ptr(d_block_hashes), hashes_cap, _stream(stream)), "smetric_route_batch_baseline")


def smetric_route_batch_sequential(idx: int, d_tokens, n_tokens: int, d_offsets, n_requests: int, d_load, w,
                                   d_instance, d_local_hit, d_global_hit, d_session_key, d_block_hashes=None,
                                   hashes_cap: int = 0, d_load_after=None, stream=None) -> None:
    _check(lib().smetric_route_batch_sequential(
        idx, _ptr(d_tokens), n_tokens, _ptr(d_offsets), n_requests, _ptr(d_load), _weights(w), _ptr(d_instance),
        _ptr(d_local_hit), _ptr(d_global_hit), _ptr(d_session_key), _ptr(d_block_hashes), hashes_cap,
        _ptr(d_load_after), _stream(stream)), "smetric_route_batch_sequential")


def smetric_reuse_workspace_bytes(n_blocks: int) -> int:
    return int(lib().smetric_reuse_workspace_bytes(n_blocks))


def smetric_reuse_breakdown(idx: int, d_tokens, n_tokens: int, d_offsets, n_requests: int, d_sessions,
                            d_sys_blocks, d_workspace, workspace_bytes: int, d_hit, d_sys, d_intra, d_inter,
                            stream=None) -> None:
    _check(lib().smetric_reuse_breakdown(idx, _ptr(d_tokens), n_tokens, _ptr(d_offsets), n_requests,
                                         _ptr(d_sessions), _ptr(d_sys_blocks), _ptr(d_workspace), workspace_bytes,
                                         _ptr(d_hit), _ptr(d_sys), _ptr(d_intra), _ptr(d_inter), _stream(stream)),
           "smetric_reuse_breakdown")


def smetric_imbalance_workspace_bytes(n_windows: int, num_instances: int) -> int:
    return int(lib().smetric_imbalance_workspace_bytes(n_windows, num_instances))


def smetric_window_imbalance(idx: int, d_instance, d_start, d_end, n_requests: int, window: int, n_windows: int,
                             d_workspace, workspace_bytes: int, d_max, d_argmax, d_sum, stream=None) -> None:
    _check(lib().smetric_window_imbalance(idx, _ptr(d_instance), _ptr(d_start), _ptr(d_end), n_requests, window,
                                          n_windows, _ptr(d_workspace), workspace_bytes, _ptr(d_max),
                                          _ptr(d_argmax), _ptr(d_sum), _stream(stream)),
           "smetric_window_imbalance")


def smetric_link_sessions(idx: int, d_tokens, n_tokens: int, d_offsets, n_requests: int, d_users, d_turns,
                          d_parent, d_session, stream=None) -> None:
    _check(lib().smetric_link_sessions(idx, _ptr(d_tokens), n_tokens, _ptr(d_offsets), n_requests, _ptr(d_users),
                                       _ptr(d_turns), _ptr(d_parent), _ptr(d_session), _stream(stream)),
           "smetric_link_sessions")


def smetric_index_commit_batch(idx: int, d_offsets, n_requests: int, d_instance, d_local_hit,
                               d_block_hashes, flags: int = 0, d_load=None, stream=None) -> None:
    _check(lib().smetric_index_commit_batch(idx, _ptr(d_offsets), n_requests, _ptr(d_instance),
                                            _ptr(d_local_hit), _ptr(d_block_hashes), flags, _ptr(d_load),
                                            _stream(stream)), "smetric_index_commit_batch")


def smetric_index_set_lru(idx: int, local_cap: int, global_cap: int) -> None:
    _check(lib().smetric_index_set_lru(idx, local_cap, global_cap), "smetric_index_set_lru")


def smetric_index_lru_sizes(idx: int, d_sizes, stream=None) -> None:
    _check(lib().smetric_index_lru_sizes(idx, _ptr(d_sizes), _stream(stream)), "smetric_index_lru_sizes")


def smetric_block_hashes(idx: int, d_tokens, n_tokens: int, d_offsets, n_requests: int,
                         d_session_key, d_block_hashes, hashes_cap: int, stream=None) -> None:
    _check(lib().smetric_block_hashes(idx, _ptr(d_tokens), n_tokens, _ptr(d_offsets), n_requests,
                                      _ptr(d_session_key), _ptr(d_block_hashes), hashes_cap,
                                      _stream(stream)), "smetric_block_hashes")


def smetric_block_hashes_noalloc(d_tokens, n_tokens: int, d_offsets, n_requests: int,
                                 block_size: int, session_blocks: int, hash_seed: int,
                                 d_session_key, d_block_hashes, hashes_cap: int, d_status,
                                 stream=None) -> int:
    """Returns the call's host-side status code (SMETRIC_ERR_TOO_LARGE for a
    batch beyond the fixed scratch); device-detected errors land in d_status."""
    return int(lib().smetric_block_hashes_noalloc(_ptr(d_tokens), n_tokens, _ptr(d_offsets), n_requests,
                                                  block_size, session_blocks, hash_seed,
                                                  _ptr(d_session_key), _ptr(d_block_hashes), hashes_cap,
                                                  _ptr(d_status), _stream(stream)))


def smetric_route_batch_host(idx: int, h_tokens, n_tokens: int, h_offsets, n_requests: int, h_load,
                             w, h_instance, h_local_hit, h_global_hit, h_session_key,
                             stream=None) -> int:
    """Returns the call's status (device-latched errors included)."""
    return int(lib().smetric_route_batch_host(idx, _ptr(h_tokens), n_tokens, _ptr(h_offsets),
                                              n_requests, _ptr(h_load), _weights(w),
                                              _ptr(h_instance), _ptr(h_local_hit),
                                              _ptr(h_global_hit), _ptr(h_session_key),
                                              _stream(stream)))


def smetric_status(idx: int, stream=None) -> int:
    return int(lib().smetric_status(idx, _stream(stream)))


def smetric_strerror(code: int) -> str:
    return lib().smetric_strerror(code).decode()


def smetric_profile_enable(idx: int, on: bool) -> None:
    _check(lib().smetric_profile_enable(idx, 1 if on else 0), "smetric_profile_enable")


def smetric_profile_read(idx: int):
    """{kernel name: (milliseconds, launches)} since the previous read."""
    ms = (C.c_double * 8)()
    ln = (C.c_int64 * 8)()
    k = lib().smetric_profile_read(idx, 8, ms, ln)
    if k < 0:
        raise SmetricError(k, "smetric_profile_read")
    return {smetric_profile_kernel_name(i): (ms[i], ln[i]) for i in range(k)}


def smetric_profile_kernel_name(k: int) -> str:
    return lib().smetric_profile_kernel_name(k).decode()


def smetric_launch_count(idx: int) -> int:
    return int(lib().smetric_launch_count(idx))


# ---------------------------------------------------------------------------
# convenience wrapper
# ---------------------------------------------------------------------------

class SMetricIndex:
    """One two-tier index on the current CUDA device, with torch outputs."""

    def __init__(self, num_instances: int, block_size: int, session_blocks: int,
                 capacity_slots: int, max_batch_requests: int, max_batch_tokens: int,
                 hash_seed: int = 0, host_staging: bool = False, pipeline: bool = False):
        self.cfg = smetric_index_config(num_instances, block_size, session_blocks,
                                        (SMETRIC_FLAG_HOST_STAGING if host_staging else 0)
                                        | (SMETRIC_FLAG_PIPELINE if pipeline else 0),
                                        capacity_slots, hash_seed & 0xFFFFFFFFFFFFFFFF,
                                        max_batch_requests, max_batch_tokens)
        self.handle = smetric_index_create(self.cfg)
        self.N, self.B, self.S = num_instances, block_size, session_blocks
        self.W = smetric_index_mask_words(self.handle)

    def close(self):
        if getattr(self, "handle", None):
            smetric_index_destroy(self.handle)
            self.handle = None

    def __enter__(self):
        return self

    def __exit__(self, *a):
        self.close()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _tiers(self, keys, tiers):
        import torch
        if isinstance(tiers, int):
            tiers = torch.full(keys.shape, tiers, dtype=torch.int32, device=keys.device)
        return tiers

    def insert(self, keys, tiers, stream=None):
        tiers = self._tiers(keys, tiers)
        smetric_index_insert(self.handle, keys, tiers, keys.numel(), stream)

    def evict(self, keys, tiers, stream=None):
        tiers = self._tiers(keys, tiers)
        smetric_index_evict(self.handle, keys, tiers, keys.numel(), stream)

    def clear(self, stream=None):
        smetric_index_clear(self.handle, stream)

    def lookup(self, keys, stream=None):
        import torch
        out = torch.empty((keys.numel(), self.W), dtype=torch.uint64, device=keys.device)
        smetric_index_lookup(self.handle, keys, keys.numel(), out, stream)
        return out

    def route_batches(self, batches, weights=(1, 4, 2), out=None, stream=None):
        """Routes a list of (tokens, offsets, load) device batches in one call;
        returns one dict(instance, local_hit, global_hit, session_key) per
        batch (or fills `out`, a list of such dicts)."""
        import torch
        if out is None:
            out = []
            for tokens, offsets, _ in batches:
                n, dev = offsets.numel() - 1, offsets.device
                out.append(dict(instance=torch.empty(n, dtype=torch.int32, device=dev),
                                local_hit=torch.empty(n, dtype=torch.int32, device=dev),
                                global_hit=torch.empty(n, dtype=torch.int32, device=dev),
                                session_key=torch.empty(n, dtype=torch.uint64, device=dev)))
        smetric_route_batches(self.handle, [b[0] for b in batches], [b[0].numel() for b in batches],
                              [b[1] for b in batches], [b[1].numel() - 1 for b in batches],
                              [b[2] for b in batches], weights, [o["instance"] for o in out],
                              [o["local_hit"] for o in out], [o["global_hit"] for o in out],
                              [o["session_key"] for o in out], stream)
        return out

    def route_batch(self, tokens, offsets, load, weights=(1, 4, 2), want_hashes=False,
                    out=None, stream=None):
        """Returns dict(instance, local_hit, global_hit, session_key[, block_hashes])."""
        import torch
        n = offsets.numel() - 1
        dev = offsets.device
        if out is None:
            out = dict(instance=torch.empty(n, dtype=torch.int32, device=dev),
                       local_hit=torch.empty(n, dtype=torch.int32, device=dev),
                       global_hit=torch.empty(n, dtype=torch.int32, device=dev),
                       session_key=torch.empty(n, dtype=torch.uint64, device=dev))
            if want_hashes:
                out["block_hashes"] = torch.empty(max(tokens.numel() // self.B, 1),
                                                  dtype=torch.uint64, device=dev)
        hb = out.get("block_hashes")
        smetric_route_batch(self.handle, tokens, tokens.numel(), offsets, n, load, weights,
                            out["instance"], out["local_hit"], out["global_hit"],
                            out["session_key"], hb, hb.numel() if hb is not None else 0, stream)
        return out

    def route_commit_batch(self, tokens, offsets, load, weights=(1, 4, 2), also_global=False, stream=None):
        """route_batch then commit_batch on the device in one call; `load` is
        read by the route and drained in place. Returns route_batch's dict
        with block_hashes."""
        import torch
        n = offsets.numel() - 1
        dev = offsets.device
        out = dict(instance=torch.empty(n, dtype=torch.int32, device=dev),
                   local_hit=torch.empty(n, dtype=torch.int32, device=dev),
                   global_hit=torch.empty(n, dtype=torch.int32, device=dev),
                   session_key=torch.empty(n, dtype=torch.uint64, device=dev),
                   block_hashes=torch.empty(max(tokens.numel() // self.B, 1), dtype=torch.uint64, device=dev))
        hb = out["block_hashes"]
        smetric_route_commit_batch(self.handle, tokens, tokens.numel(), offsets, n, load, weights, out["instance"],
                                   out["local_hit"], out["global_hit"], out["session_key"], hb, hb.numel(),
                                   SMETRIC_COMMIT_GLOBAL if also_global else 0, stream)
        return out

    def route_batch_policy(self, tokens, offsets, queued, turn, est_hit, policy, want_hashes=False,
                           out=None, stream=None):
        """The session-centric policy (Figure 10). `policy` is a dict with c_lin,
        c_att, ttft_d0, ttft_d1, hit_num, hit_den and optionally rr_base.
        Returns dict(instance, local_hit, global_hit, stick, session_key[, block_hashes])."""
        import torch
        n = offsets.numel() - 1
        dev = offsets.device
        if out is None:
            out = dict(instance=torch.empty(n, dtype=torch.int32, device=dev),
                       local_hit=torch.empty(n, dtype=torch.int32, device=dev),
                       global_hit=torch.empty(n, dtype=torch.int32, device=dev),
                       stick=torch.empty(n, dtype=torch.int32, device=dev),
                       session_key=torch.empty(n, dtype=torch.uint64, device=dev))
            if want_hashes:
                out["block_hashes"] = torch.empty(max(tokens.numel() // self.B, 1),
                                                  dtype=torch.uint64, device=dev)
        hb = out.get("block_hashes")
        smetric_route_batch_policy(self.handle, tokens, tokens.numel(), offsets, n, queued, turn, est_hit,
                                   policy, out["instance"], out["local_hit"], out["global_hit"],
                                   out["stick"], out["session_key"], hb,
                                   hb.numel() if hb is not None else 0, stream)
        return out

    def route_batch_policy_coloc(self, tokens, offsets, queued, tpot_budget, num_requests, turn, est_hit,
                                 policy, want_hashes=False, stream=None):
        """The session-centric policy under PD colocation (Appendix B).
        Returns dict(instance, local_hit, global_hit, stick, session_key[, block_hashes])."""
        import torch
        n = offsets.numel() - 1
        dev = offsets.device
        out = dict(instance=torch.empty(n, dtype=torch.int32, device=dev),
                   local_hit=torch.empty(n, dtype=torch.int32, device=dev),
                   global_hit=torch.empty(n, dtype=torch.int32, device=dev),
                   stick=torch.empty(n, dtype=torch.int32, device=dev),
                   session_key=torch.empty(n, dtype=torch.uint64, device=dev))
        if want_hashes:
            out["block_hashes"] = torch.empty(max(tokens.numel() // self.B, 1), dtype=torch.uint64, device=dev)
        hb = out.get("block_hashes")
        smetric_route_batch_policy_coloc(self.handle, tokens, tokens.numel(), offsets, n, queued, tpot_budget,
                                         num_requests, turn, est_hit, policy, out["instance"], out["local_hit"],
                                         out["global_hit"], out["stick"], out["session_key"], hb,
                                         hb.numel() if hb is not None else 0, stream)
        return out

    def route_batch_baseline(self, tokens, offsets, scorer, queued, batch, lam=(1, 2), stream=None):
        """A baseline scorer of Section 5.1 (SMETRIC_SCORER_BAILIAN or _LMETRIC).
        Returns dict(instance, local_hit, global_hit, session_key)."""
        import torch
        n = offsets.numel() - 1
        dev = offsets.device
        out = dict(instance=torch.empty(n, dtype=torch.int32, device=dev),
                   local_hit=torch.empty(n, dtype=torch.int32, device=dev),
                   global_hit=torch.empty(n, dtype=torch.int32, device=dev),
                   session_key=torch.empty(n, dtype=torch.uint64, device=dev))
        smetric_route_batch_baseline(self.handle, tokens, tokens.numel(), offsets, n, scorer, queued, batch,
                                     lam[0], lam[1], out["instance"], out["local_hit"], out["global_hit"],
                                     out["session_key"], None, 0, stream)
        return out

    def route_batch_sequential(self, tokens, offsets, load, weights=(1, 4, 2), stream=None):
        """The argmin cost with loads updated request by request. Returns
        dict(instance, local_hit, global_hit, session_key, load_after)."""
        import torch
        n = offsets.numel() - 1
        dev = offsets.device
        out = dict(instance=torch.empty(n, dtype=torch.int32, device=dev),
                   local_hit=torch.empty(n, dtype=torch.int32, device=dev),
                   global_hit=torch.empty(n, dtype=torch.int32, device=dev),
                   session_key=torch.empty(n, dtype=torch.uint64, device=dev),
                   load_after=torch.empty(self.N, dtype=torch.int64, device=dev))
        smetric_route_batch_sequential(self.handle, tokens, tokens.numel(), offsets, n, load, weights,
                                       out["instance"], out["local_hit"], out["global_hit"], out["session_key"],
                                       None, 0, out["load_after"], stream)
        return out

    def reuse_breakdown(self, tokens, offsets, sessions, sys_blocks, workspace=None, stream=None):
        """KV$ reuse against an unbounded store of the earlier requests:
        dict(hit, sys, intra, inter), int32 blocks per request."""
        import torch
        n = offsets.numel() - 1
        dev = offsets.device
        need = smetric_reuse_workspace_bytes(tokens.numel() // self.B)
        if workspace is None:
            workspace = torch.empty(need, dtype=torch.uint8, device=dev)
        out = {k: torch.empty(n, dtype=torch.int32, device=dev) for k in ("hit", "sys", "intra", "inter")}
        smetric_reuse_breakdown(self.handle, tokens, tokens.numel(), offsets, n, sessions, sys_blocks, workspace,
                                workspace.numel(), out["hit"], out["sys"], out["intra"], out["inter"], stream)
        return out

    def window_imbalance(self, instance, start, end, window: int, n_windows: int, workspace=None, stream=None):
        """Per window: dict(max, argmax, sum) of the instances' running-request
        ticks; the imbalance is N * max / sum."""
        import torch
        dev = start.device
        if workspace is None:
            workspace = torch.empty(max(1, smetric_imbalance_workspace_bytes(n_windows, self.N) // 8),
                                    dtype=torch.int64, device=dev)
        out = dict(max=torch.empty(n_windows, dtype=torch.int64, device=dev),
                   argmax=torch.empty(n_windows, dtype=torch.int32, device=dev),
                   sum=torch.empty(n_windows, dtype=torch.int64, device=dev))
        smetric_window_imbalance(self.handle, instance, start, end, instance.numel(), window, n_windows, workspace,
                                 workspace.numel() * workspace.element_size(), out["max"], out["argmax"],
                                 out["sum"], stream)
        return out

    def link_sessions(self, tokens, offsets, users, turns, stream=None):
        """Session reconstruction (Appendix A): returns (parent, session), int32 per request."""
        import torch
        n = offsets.numel() - 1
        parent = torch.empty(n, dtype=torch.int32, device=offsets.device)
        session = torch.empty(n, dtype=torch.int32, device=offsets.device)
        smetric_link_sessions(self.handle, tokens, tokens.numel(), offsets, n, users, turns, parent, session,
                              stream)
        return parent, session

    def commit_batch(self, offsets, out, also_global=False, load=None, stream=None):
        """Add the routed batch's blocks (`out` from route_batch(..., want_hashes=True)
        or route_batch_policy) to its chosen instances' local tiers (and the
        global tier); with `load`, drain it in place."""
        smetric_index_commit_batch(self.handle, offsets, offsets.numel() - 1, out["instance"],
                                   out["local_hit"], out["block_hashes"],
                                   SMETRIC_COMMIT_GLOBAL if also_global else 0, load, stream)

    def set_lru(self, local_cap=0, global_cap=0):
        """Caps the local tiers at `local_cap` blocks each and the global tier
        at `global_cap` (0: uncapped); commit_batch then evicts each capped
        tier's least recently used blocks on the device."""
        smetric_index_set_lru(self.handle, int(local_cap), int(global_cap))

    def lru_sizes(self, stream=None):
        """Blocks the device LRU tracks per tier (int64 [N+1], global last)."""
        import torch
        out = torch.empty(self.N + 1, dtype=torch.int64, device="cuda")
        smetric_index_lru_sizes(self.handle, out, stream)
        return out

    def block_hashes(self, tokens, offsets, stream=None):
        """Returns (block_hashes, session_key) as device tensors."""
        import torch
        n = offsets.numel() - 1
        dev = offsets.device
        hb = torch.empty(max(tokens.numel() // self.B, 1), dtype=torch.uint64, device=dev)
        sk = torch.empty(max(n, 1), dtype=torch.uint64, device=dev)
        smetric_block_hashes(self.handle, tokens, tokens.numel(), offsets, n, sk, hb, hb.numel(),
                             stream)
        return hb, sk[:n]

    def status(self, stream=None) -> int:
        return smetric_status(self.handle, stream)

    def check(self, stream=None):
        rc = self.status(stream)
        if rc != SMETRIC_OK:
            raise SmetricError(rc, "device")
