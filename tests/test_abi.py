"""The C-ABI library loads and exports every symbol include/smetric.h
declares; host-side argument checks reject bad input before any CUDA call
(no GPU needed)."""

import ctypes as C
import os
import re

import pytest

import paper_2607_08565_gb300 as pkg
from paper_2607_08565_gb300 import build_lib

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    src = open(os.path.join(ROOT, "include", "smetric.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(smetric_[a-z_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def L():
    build_lib.build()
    return pkg.lib()


def test_header_declares_the_binding_names():
    assert _declared() == sorted(pkg.EXPORTED)


def test_library_exports_every_declared_symbol(L):
    for name in _declared():
        assert hasattr(L, name), name


def test_library_links_no_python_or_torch():
    import subprocess
    out = subprocess.run(["ldd", build_lib.LIB], capture_output=True, text=True).stdout
    assert "torch" not in out and "python" not in out


def test_strerror_and_kernel_names(L):
    assert pkg.smetric_strerror(pkg.SMETRIC_ERR_TABLE_FULL) == "index table full"
    assert pkg.smetric_strerror(12345) == "unknown error"
    assert [pkg.smetric_profile_kernel_name(k) for k in range(4)] == ["k_prep", "k_digest", "k_chain_probe",
                                                                      "k_walk"]
    assert pkg.smetric_profile_kernel_name(4) == ""


def _create(L, **kw):
    base = dict(num_instances=4, block_size=16, session_blocks=2, flags=0, capacity_slots=64,
                hash_seed=0, max_batch_requests=8, max_batch_tokens=1024)
    base.update(kw)
    cfg = pkg.smetric_index_config(**base)
    h = C.c_void_p()
    return L.smetric_index_create(C.byref(cfg), C.byref(h)), h.value


@pytest.mark.parametrize("bad", [
    dict(num_instances=0), dict(num_instances=257), dict(block_size=7), dict(block_size=0),
    dict(block_size=258), dict(session_blocks=0), dict(capacity_slots=0),
    dict(max_batch_requests=-1), dict(max_batch_tokens=-5), dict(flags=8), dict(flags=4),
    dict(capacity_slots=(1 << 64) - 1),
])
def test_create_rejects_bad_config_on_host(L, bad):
    rc, h = _create(L, **bad)
    assert rc == pkg.SMETRIC_ERR_INVALID_ARG and not h


def test_binding_constants_match_the_header():
    """Every #define SMETRIC_* value in the header equals the binding's."""
    text = open(os.path.join(ROOT, "include", "smetric.h")).read()
    seen = 0
    for name, expr in re.findall(r"^#define (SMETRIC_\w+) ([^/\n]+)", text, re.M):
        if name == "SMETRIC_H":
            continue
        value = eval(expr.replace("LL", "").strip(), {})
        assert getattr(pkg, name) == value, name
        seen += 1
    assert seen >= 15


def test_workspace_sizes(L):
    # the reuse table: 16-byte slots for twice the blocks (a power of two, at least 64) and a 32-byte header
    assert L.smetric_reuse_workspace_bytes(0) == 16 * 64 + 32
    assert L.smetric_reuse_workspace_bytes(1000) == 16 * 2048 + 32
    assert L.smetric_reuse_workspace_bytes(1024) == 16 * 2048 + 32
    assert L.smetric_reuse_workspace_bytes(-1) == 0
    # the imbalance grid: one int64 per (window, instance)
    assert L.smetric_imbalance_workspace_bytes(30, 32) == 8 * 30 * 32
    assert L.smetric_imbalance_workspace_bytes(-1, 32) == 0


def test_null_handles_are_rejected(L):
    assert L.smetric_index_create(None, None) == pkg.SMETRIC_ERR_INVALID_ARG
    assert L.smetric_index_destroy(None) == pkg.SMETRIC_OK
    assert L.smetric_index_insert(None, None, None, 0, None) == pkg.SMETRIC_ERR_INVALID_ARG
    assert L.smetric_route_batch(None, None, 0, None, 0, None, pkg.smetric_weights(1, 4, 2),
                                 None, None, None, None, None, 0, None) == pkg.SMETRIC_ERR_INVALID_ARG
    assert L.smetric_route_batch_policy(None, None, 0, None, 0, None, None, None,
                                        pkg.smetric_policy(1, 1, 0, 0, 1, 2, 0, 0), None, None, None,
                                        None, None, None, 0, None) == pkg.SMETRIC_ERR_INVALID_ARG
    assert L.smetric_status(None, None) == pkg.SMETRIC_ERR_INVALID_ARG
    assert L.smetric_reuse_breakdown(None, None, 0, None, 1, None, None, None, 0, None, None, None, None,
                                     None) == pkg.SMETRIC_ERR_INVALID_ARG
    assert L.smetric_window_imbalance(None, None, None, None, 0, 1, 1, None, 0, None, None, None,
                                      None) == pkg.SMETRIC_ERR_INVALID_ARG
    w = pkg.smetric_weights(1, 4, 2)
    assert L.smetric_route_batches(None, 0, None, None, None, None, None, w, None, None, None, None,
                                   None) == pkg.SMETRIC_ERR_INVALID_ARG
    assert L.smetric_index_mask_words(None) == 0
    assert L.smetric_launch_count(None) == 0


def test_noalloc_hashes_refuse_on_host(L):
    """Refusals of smetric_block_hashes_noalloc that need no device: a batch
    beyond its fixed scratch, a bad block size, an empty batch (a no-op)."""
    f = L.smetric_block_hashes_noalloc
    assert f(None, 0, None, pkg.SMETRIC_NOALLOC_MAX_REQUESTS + 1, 16, 1, 0, None, None, 0, None,
             None) == pkg.SMETRIC_ERR_TOO_LARGE
    assert f(None, 16 * (pkg.SMETRIC_NOALLOC_MAX_BLOCKS + 1), None, 1, 16, 1, 0, None, None, 0, None,
             None) == pkg.SMETRIC_ERR_TOO_LARGE
    assert f(None, 0, None, 1, 7, 1, 0, None, None, 0, None, None) == pkg.SMETRIC_ERR_INVALID_ARG
    assert f(None, 0, None, 1, 16, 0, 0, None, None, 0, None, None) == pkg.SMETRIC_ERR_INVALID_ARG
    assert f(None, 0, None, 0, 16, 1, 0, None, None, 0, None, None) == pkg.SMETRIC_OK
    assert pkg.smetric_strerror(pkg.SMETRIC_ERR_TOO_LARGE) == \
        "batch larger than the fixed no-allocation scratch"


def test_header_is_plain_c_and_matches_the_binding_layout(tmp_path, L):
    """include/smetric.h compiles as strict C99 with no CUDA header, links
    against libsmetric.so, and its structs and enum agree byte for byte with
    the ctypes binding; the refusals it makes from C need no GPU."""
    import shutil
    import subprocess
    if shutil.which("gcc") is None:
        pytest.skip("no C compiler")
    exe = str(tmp_path / "c_abi_check")
    libdir = os.path.dirname(build_lib.LIB)
    subprocess.check_call(["gcc", "-std=c99", "-pedantic", "-Wall", "-Wextra", "-Werror",
                           "-I", os.path.join(ROOT, "include"), os.path.join(ROOT, "tests", "c_abi_check.c"),
                           "-o", exe, "-L", libdir, "-lsmetric", "-Wl,-rpath," + libdir])
    out = subprocess.run([exe], capture_output=True, text=True, check=True).stdout.splitlines()
    structs = {"smetric_index_config": pkg.smetric_index_config, "smetric_weights": pkg.smetric_weights,
               "smetric_policy": pkg.smetric_policy}
    fields = 0
    for line in out:
        kind, *rest = line.split(" ", 1)
        rest = rest[0] if rest else ""
        if kind == "sizeof":
            name, size = rest.split()
            assert C.sizeof(structs[name]) == int(size), name
        elif kind == "offset":
            qual, off, size = rest.split()
            name, field = qual.split(".")
            desc = getattr(structs[name], field)
            assert (desc.offset, desc.size) == (int(off), int(size)), qual
            fields += 1
        elif kind == "enum":
            name, value = rest.split()
            assert getattr(pkg, name) == int(value), name
        elif kind == "call":
            what, *vals = rest.split()
            want = {"create_odd_block": [pkg.SMETRIC_ERR_INVALID_ARG, 1],
                    "route_null_index": [pkg.SMETRIC_ERR_INVALID_ARG],
                    "destroy_null": [pkg.SMETRIC_OK]}[what]
            assert [int(v) for v in vals] == want, what
        elif kind == "strerror":
            assert rest == pkg.smetric_strerror(pkg.SMETRIC_ERR_TABLE_FULL)
    assert fields == 8 + 3 + 8
    # every struct field of the binding was printed by the C side
    assert fields == sum(len(s._fields_) for s in structs.values())
